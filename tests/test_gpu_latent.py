"""GPU parity of the latent form (one bottleneck c = h W_down per token
shared by every head, keys and values; Sec. 2 Eq. 1-4 with the cache scheme
of Sec. 5) against the CPU oracle, through the C ABI: dar_latent_append (the
cached bottleneck, bit-exact), dar_latent_absorb and dar_latent_decode
(max-abs 2e-2, bf16 storage with fp32 accumulation)."""
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

TOL = 2e-2


def check_decode(wl, seqs, heads_of):
    cfg = wl.cfg
    out = wl.decode()
    torch.cuda.synchronize()
    assert wl.cache.device_status() == 0
    got = W.to_f64(W.download(out), "bf16")
    assert np.isfinite(got).all()
    k, v, h = wl.history_arrays(seqs)
    Wdown, Wup, WK, WV = wl.proj_host
    heads = [(i, hq) for i, b in enumerate(seqs) for hq in heads_of(b)]
    want = oracle.latent_decode(np.ascontiguousarray(wl.q_host[seqs]), k, v, h, wl.lens[seqs], Wdown, Wup, WK, WV,
                                cfg.w, "bf16", heads=heads)
    err = max(np.abs(got[seqs[i], hq] - want[i, hq]).max() for i, hq in heads)
    assert err <= TOL, err


def test_latent_160m_decode():
    """B32 H12 L4096 D768 d_lat 192 w128: one head of every sequence, every
    head of three sequences."""
    cfg = I.DECODE_160M_LATENT
    wl = W.LatentDecodeWorkload(cfg, keep_history=True)
    seqs = list(range(cfg.B))
    check_decode(wl, seqs, lambda b: range(cfg.Hq) if b in (0, 13, 31) else [(5 * b) % cfg.Hq])


def test_latent_1b_gqa_decode():
    """B64 Hq32 Hkv8 D2048 d_lat 256 w256, ragged lengths, shuffled pages: the
    query heads of one KV head in eight sequences (shortest, longest, others)."""
    cfg = I.DECODE_1B_LATENT
    wl = W.LatentDecodeWorkload(cfg, keep_history=True)
    lens = wl.lens
    seqs = sorted({int(np.argmin(lens)), int(np.argmax(lens)), 0, 9, 22, 37, 50, 63})
    G = cfg.Hq // cfg.Hkv
    check_decode(wl, seqs, lambda b: [G * (b % cfg.Hkv) + j for j in range(G)])


SMALL = [
    # B, Hq, Hkv, D, d_lat, w, L range
    (5, 4, 2, 96, 64, 40, (1, 300)),      # ragged around the window, empty-ish latent parts
    (3, 16, 16, 128, 128, 64, (64, 65)),  # L = w and w + 1
    (4, 32, 8, 64, 192, 1, (250, 700)),   # only the current token local
    (2, 8, 1, 256, 256, 300, (700, 1100)),
]


@pytest.mark.parametrize("case", SMALL, ids=lambda c: "-".join(map(str, c[:6])))
def test_latent_small_cases(case):
    B, Hq, Hkv, D, dl, w, rng = case
    cfg = I.LatentDecode("latent case", 300 + D + dl + w, B, Hq, Hkv, 64, D, dl, w, L_range=rng, shuffle_pages=True)
    wl = W.LatentDecodeWorkload(cfg, keep_history=True, chunk=97)
    check_decode(wl, list(range(B)), lambda b: range(Hq))


def test_latent_append_is_exact():
    """The cached bottleneck equals Eq. 1 (oracle chain over D) bit for bit,
    token-by-token appends equal one bulk append, and the ring holds the last
    w keys/values."""
    cfg = I.LatentDecode("latent append", 77, 3, 4, 2, 64, 160, 64, 24, L_range=(10, 150), shuffle_pages=True)
    bulk = W.LatentDecodeWorkload(cfg, keep_history=True, chunk=1000)
    step = W.LatentDecodeWorkload(cfg, keep_history=False, chunk=1)
    assert bulk.cache.device_status() == 0 and step.cache.device_status() == 0
    Wdown = bulk.proj_host[0]
    table = bulk.cache.block_table.cpu().numpy()
    pool = W.download(bulk.cache.pool_c)
    assert np.array_equal(pool, W.download(step.cache.pool_c))
    for name in ("win_k", "win_v", "seq_lens"):
        assert torch.equal(getattr(bulk.cache, name), getattr(step.cache, name)), name
    for b in range(cfg.B):
        L = int(bulk.lens[b])
        h, k, v = bulk.history[b]
        c = oracle.latent_bottleneck(h[None], Wdown, "bf16")[0]
        rows = np.stack([pool[table[b, p // 64], p % 64] for p in range(L)])
        assert np.array_equal(rows, c)
        win = W.download(bulk.cache.win_k)[b]
        for p in range(max(0, L - cfg.w), L):
            assert np.array_equal(win[:, p % cfg.w], k[:, p])


def test_latent_absorb_matches_products():
    """A_K = W_up W_K and A_V = W_up W_V per KV head (fp32 chains; compared with
    float64 products at fp32 accuracy)."""
    Wdown, Wup, WK, WV = I.latent_projections(5, 3, 512, 128, 64)
    A_K, A_V = dar.dar_latent_absorb(*(W.upload(x, "f32") for x in (Wup, WK, WV)))
    for A, M, spec in ((A_K, WK, "ce,get->gtc"), (A_V, WV, "ce,get->gct")):  # A_K is stored transposed
        want = np.einsum(spec, Wup.astype(np.float64), M.astype(np.float64))
        np.testing.assert_allclose(A.cpu().numpy(), want, rtol=0, atol=2e-5)
