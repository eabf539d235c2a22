"""GPU decode parity against the CPU oracle (through the C ABI), on caches
filled by dar_cache_append.  bf16 tolerance 2e-2 max-abs, fp32 1e-5."""
import numpy as np
import pytest

import oracle
from paper_2606_18587_gb300 import inputs as I

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("no CUDA device", allow_module_level=True)

from paper_2606_18587_gb300 import dar  # noqa: E402
from paper_2606_18587_gb300 import workloads as W  # noqa: E402

TOL = {"f32": 1e-5, "bf16": 2e-2}


def oracle_decode(wl, heads=None, lens=None):
    k, v = wl.history_arrays()
    Dk, Uk, Dv, Uv = wl.proj_host
    lens = wl.lens if lens is None else lens
    return oracle.decode(wl.q_host, k, v, lens, Dk, Uk, Dv, Uv, wl.cfg.w, wl.cfg.dtype, heads=heads)


def gpu_out(wl):
    out = wl.decode()
    torch.cuda.synchronize()
    assert wl.cache.device_status() == 0
    return W.to_f64(W.download(out), wl.cfg.dtype)


def test_decode_160m_all_heads():
    """B32 H12 L4096 d64 dd16 w128 bf16: every (b, h)."""
    wl = W.DecodeWorkload(I.DECODE_160M, keep_history=True)
    got = gpu_out(wl)
    want = oracle_decode(wl)
    err = np.abs(got - want).max()
    assert err <= TOL["bf16"], err


def test_decode_160m_repeat_calls_identical():
    """The workspace resets itself: repeated calls give bit-identical outputs."""
    wl = W.DecodeWorkload(I.DECODE_160M)
    a = W.download(wl.decode()).copy()
    for _ in range(3):
        b = W.download(wl.decode())
    np.testing.assert_array_equal(a, b)


def test_decode_1b_gqa_paged():
    """B64 Hq32 Hkv8 dd16 w256, ragged L in [1024, 32768], shuffled 64-token
    pages; the oracle checks one head of every sequence (cycling through the
    heads) and every head of the shortest, the longest and a few others."""
    cfg = I.DECODE_1B_GQA
    wl = W.DecodeWorkload(cfg, keep_history=True)
    got = gpu_out(wl)
    lens = wl.lens
    seqs = sorted({int(np.argmin(lens)), int(np.argmax(lens)), 0, 17, 42})
    heads = sorted({(b, h) for b in seqs for h in range(cfg.Hq)} | {(b, (5 * b) % cfg.Hq) for b in range(cfg.B)})
    want = oracle_decode(wl, heads=heads)
    err = max(np.abs(got[b, h] - want[b, h]).max() for b, h in heads)
    assert err <= TOL["bf16"], err
    assert np.isfinite(got).all()


@pytest.mark.parametrize("k", range(16))
def test_decode_sweep_point(k):
    """B16 H16 L16384, w in {64, 256, 1024, 16384} x d_down in {8, 16, 32, 64}:
    one head of every sequence, and every head of the first and last
    (w = 16384 is plain attention)."""
    cfg = I.sweep_point(k)
    wl = W.DecodeWorkload(cfg, keep_history=True)
    got = gpu_out(wl)
    heads = sorted({(b, h) for b in (0, cfg.B - 1) for h in range(cfg.Hq)} | {(b, (3 * b + k) % cfg.Hq)
                                                                           for b in range(cfg.B)})
    want = oracle_decode(wl, heads=heads)
    err = max(np.abs(got[b, h] - want[b, h]).max() for b, h in heads)
    assert err <= TOL["bf16"], err
    assert np.isfinite(got).all()


SMALL = [
    # dtype, B, Hq, Hkv, dd, w, lens
    ("f32", 3, 4, 4, 16, 32, [1, 31, 500]),
    ("f32", 2, 8, 2, 64, 7, [64, 1000]),
    ("bf16", 4, 6, 2, 8, 1, [1, 2, 65, 129]),      # only the current token is local
    ("bf16", 3, 8, 1, 32, 300, [299, 300, 301]),   # window edge, MQA (G = 8)
    ("bf16", 2, 3, 3, 16, 64, [0, 77]),            # an empty sequence gets zeros
]


@pytest.mark.parametrize("case", SMALL, ids=lambda c: "-".join(map(str, c[:6])))
def test_decode_small_cases(case):
    dtype, B, Hq, Hkv, dd, w, lens = case
    cfg = I.Decode("small", 90 + dd + w, B, Hq, Hkv, 64, dd, w, dtype, L_range=(1, 2), shuffle_pages=True)
    wl = W.DecodeWorkload(cfg, keep_history=True, lens=np.array(lens))
    got = gpu_out(wl)
    want = oracle_decode(wl)
    err = np.abs(got - want).max()
    assert err <= TOL[dtype], err
    for b, L in enumerate(lens):
        if L == 0:
            assert np.all(got[b] == 0)


def test_decode_identity_bottleneck_is_full_attention():
    """d_down = d with identity projections: the cached vectors equal the keys
    and values, so the output equals plain causal attention (oracle with w >= L)."""
    cfg = I.Decode("identity", 95, 2, 4, 4, 64, 64, 16, "f32", L_range=(1, 2))
    wl = W.DecodeWorkload(cfg, keep_history=True, lens=np.array([40, 300]))
    eye = torch.eye(64, dtype=torch.float32, device="cuda").expand(4, 64, 64).contiguous()
    # a second cache over the same history, filled with identity down-projections
    cache = dar.DarCache(2, 4, 64, 16, wl.cache.max_pages_per_seq, wl.cache.num_pages, dtype=torch.float32,
                         block_table=wl.cache.block_table.cpu())
    k, v = wl.history_arrays()
    counts = torch.tensor([40, 300], dtype=torch.int32, device="cuda")
    dar.dar_cache_append(cache, W.upload(k, "f32"), W.upload(v, "f32"), eye, eye, n_per_seq=counts)
    out = dar.dar_attn_decode(cache, wl.q, eye, eye, dar.decode_workspace(cache, 4))
    torch.cuda.synchronize()
    got = W.download(out).astype(np.float64)
    ident = np.broadcast_to(np.eye(64, dtype=np.float32), (4, 64, 64)).copy()
    want = oracle.decode(wl.q_host, k, v, wl.lens, ident, ident, ident, ident, 10 ** 6, "f32")
    assert np.abs(got - want).max() <= TOL["f32"]


def test_page_permutation_bit_identical():
    """Physical page placement does not change a single output bit."""
    lens = np.array([700, 1500, 64])
    base = I.Decode("perm", 96, 3, 4, 2, 64, 16, 64, "bf16", L_range=(1, 2), shuffle_pages=False)
    shuf = I.Decode("perm", 96, 3, 4, 2, 64, 16, 64, "bf16", L_range=(1, 2), shuffle_pages=True)
    a = W.DecodeWorkload(base, lens=lens)
    b = W.DecodeWorkload(shuf, lens=lens)
    assert not np.array_equal(a.table, b.table)
    np.testing.assert_array_equal(W.download(a.decode()), W.download(b.decode()))


def test_decode_steps_follow_prefill_rows():
    """Token-by-token: after appending tokens 0..t, decode with query q_t gives
    prefill row t (both within tolerance of the oracle and of each other)."""
    cfg = I.Prefill("steps", 97, 1, 4, 2, 150, 64, 16, 40, "bf16")
    pw = W.PrefillWorkload(cfg)
    pw.run()
    pre = W.to_f64(W.download(pw.out), "bf16")
    cache = dar.DarCache(1, 2, 16, 40, 2, 2, dtype=torch.bfloat16)
    ws = dar.decode_workspace(cache, 4)
    for t in range(cfg.N):
        dar.dar_cache_append(cache, pw.k[:, :, t:t + 1].contiguous(), pw.v[:, :, t:t + 1].contiguous(), pw.Dk, pw.Dv)
        if t in (0, 1, 38, 39, 40, 41, 64, 100, 149):
            out = dar.dar_attn_decode(cache, pw.q[:, :, t].contiguous(), pw.Uk, pw.Uv, ws)
            got = W.to_f64(W.download(out), "bf16")
            assert np.abs(got[0] - pre[0, :, t]).max() <= 2e-2
    torch.cuda.synchronize()
    assert cache.device_status() == 0
