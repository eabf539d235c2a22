"""Chunked prefill over an existing cache (dar_prefill_chunk) against the CPU
oracle: the chunk's output rows equal the causal forward over the whole
sequence at positions L_b .. L_b + n - 1, and the cache afterwards is
bit-identical to n one-token appends.  bf16 tolerance 2e-2 max-abs."""
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


def _chunk_inputs(cfg, n, seed):
    q = I.normal_array(seed, I.S_Q, (cfg.B, cfg.Hq, n, cfg.d), dtype=cfg.dtype)
    k = I.normal_array(seed, I.S_K, (cfg.B, cfg.Hkv, n, cfg.d), dtype=cfg.dtype)
    v = I.normal_array(seed, I.S_V, (cfg.B, cfg.Hkv, n, cfg.d), dtype=cfg.dtype)
    return q, k, v


def _oracle_rows(wl, q, k, v):
    """Oracle rows L_b .. L_b + n - 1 of the whole sequence, per sequence."""
    cfg = wl.cfg
    n = q.shape[2]
    hk, hv = wl.history_arrays() if wl.history else (None, None)
    Dk, Uk, Dv, Uv = wl.proj_host
    out = np.zeros(q.shape, dtype=np.float64)
    for b in range(cfg.B):
        L = int(wl.lens[b])
        kk = np.zeros((1, cfg.Hkv, L + n, cfg.d), dtype=q.dtype)
        vv = np.zeros_like(kk)
        if L:
            kk[0, :, :L], vv[0, :, :L] = hk[b, :, :L], hv[b, :, :L]
        kk[0, :, L:], vv[0, :, L:] = k[b], v[b]
        qq = np.zeros((1, cfg.Hq, L + n, cfg.d), dtype=q.dtype)
        qq[0, :, L:] = q[b]
        rows = np.array([(0, h, L + r) for h in range(cfg.Hq) for r in range(n)])
        res = oracle.prefill(qq, kk, vv, Dk, Uk, Dv, Uv, cfg.w, cfg.dtype, rows=rows)
        out[b] = res.reshape(cfg.Hq, n, cfg.d)
    return out


CASES = [
    # B, Hq, Hkv, dd, w, lens, n
    (3, 4, 2, 16, 64, [300, 1000, 64], 96),     # window edge inside the chunk, ragged lengths
    (2, 2, 2, 16, 37, [0, 500], 130),           # an empty cache (plain prefill), chunk over 128 rows
    (2, 8, 2, 32, 128, [1, 2000], 200),         # G = 4, d_down 32
    (1, 2, 1, 64, 16, [700], 40),               # d_down 64, short window
    (2, 2, 2, 16, 1, [129, 64], 70),            # only the current token is local
    (2, 4, 4, 16, 512, [40, 3000], 256),        # the 410M-like window
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "-".join(str(x) for x in (c[0], c[1], c[2], c[3], c[4], c[6])))
def test_chunk_matches_oracle_and_token_by_token_cache(case):
    B, Hq, Hkv, dd, w, lens, n = case
    cfg = I.Decode("chunk", 150 + dd + w + n, B, Hq, Hkv, 64, dd, w, "bf16", L_range=(1, 2), shuffle_pages=True)
    lens = np.array(lens)
    wl = W.DecodeWorkload(cfg, extra_tokens=n, keep_history=True, lens=lens)
    ref = W.DecodeWorkload(cfg, extra_tokens=n, lens=lens)  # the same cache, appended token by token
    q, k, v = _chunk_inputs(cfg, n, 160 + n)
    qd, kd, vd = W.upload(q, "bf16"), W.upload(k, "bf16"), W.upload(v, "bf16")
    out = dar.dar_prefill_chunk(wl.cache, qd, kd, vd, wl.Dk, wl.Uk, wl.Dv, wl.Uv)
    for t in range(n):
        dar.dar_cache_append(ref.cache, kd[:, :, t:t + 1].contiguous(), vd[:, :, t:t + 1].contiguous(), ref.Dk, ref.Dv)
    torch.cuda.synchronize()
    assert wl.cache.device_status() == 0 and ref.cache.device_status() == 0
    got = W.to_f64(W.download(out), "bf16")
    assert np.isfinite(got).all()
    want = _oracle_rows(wl, q, k, v)
    err = np.abs(got - want).max()
    assert err <= TOL, err
    for name in ("win_k", "win_v", "pool_kd", "pool_vd", "seq_lens"):
        np.testing.assert_array_equal(W.download(getattr(wl.cache, name)), W.download(getattr(ref.cache, name)),
                                      err_msg=name)


def test_chunks_follow_the_whole_prefill():
    """A prompt entered in four chunks gives the rows of one prefill over the
    whole sequence."""
    cfg = I.Prefill("chunks", 171, 1, 4, 2, 600, 64, 16, 100, "bf16")
    pw = W.PrefillWorkload(cfg)
    pw.run()
    full = W.to_f64(W.download(pw.out), "bf16")
    cache = dar.DarCache(1, 2, 16, 100, 10, 10, dtype=torch.bfloat16)
    cuts = [0, 150, 310, 590, 600]
    for a, b in zip(cuts[:-1], cuts[1:]):
        sl = slice(a, b)
        q = pw.q[:, :, sl].contiguous()
        out = dar.dar_prefill_chunk(cache, q, pw.k[:, :, sl].contiguous(), pw.v[:, :, sl].contiguous(), pw.Dk,
                                    pw.Uk, pw.Dv, pw.Uv)
        got = W.to_f64(W.download(out), "bf16")
        assert np.abs(got[0] - full[0, :, sl]).max() <= TOL
    torch.cuda.synchronize()
    assert cache.device_status() == 0
    assert int(W.download(cache.seq_lens)[0]) == 600


def test_chunk_rejects_unsupported_shapes():
    cache = dar.DarCache(1, 2, 8, 16, 2, 2, dtype=torch.bfloat16)  # d_down 8 is not built for chunks
    q = torch.zeros((1, 2, 4, 64), dtype=torch.bfloat16, device="cuda")
    kv = torch.zeros((1, 2, 4, 64), dtype=torch.bfloat16, device="cuda")
    D = torch.zeros((2, 64, 8), dtype=torch.float32, device="cuda")
    U = torch.zeros((2, 8, 64), dtype=torch.float32, device="cuda")
    with pytest.raises(dar.DarError) as e:
        dar.dar_prefill_chunk(cache, q, kv, kv, D, U, D, U)
    assert e.value.code == dar.DAR_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert int(W.download(cache.seq_lens)[0]) == 0  # nothing appended
