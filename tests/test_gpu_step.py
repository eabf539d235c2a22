"""The serving step (dar_decode_step: append + decode with the decode's query
set-up overlapping the append) against the oracle, eagerly and captured in a
CUDA graph with the same launch edges the benchmark times, plus the ordering
contract of dar_attn_decode.  bf16 tolerance 2e-2 max-abs."""
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


def _steps(cfg, nsteps):
    """Per-step new tokens and queries (host arrays) of a decode workload."""
    toks = [I.decode_new_tokens(cfg, s) for s in range(nsteps)]
    qs = [I.decode_query(cfg, step=s + 1) for s in range(nsteps)]
    return toks, qs


def _oracle_after(wl, toks, qs, nsteps):
    """Oracle decode of the last step: history + the appended tokens."""
    k, v = wl.history_arrays()
    cfg = wl.cfg
    lens = wl.lens + nsteps
    Lmax = int(lens.max())
    k2 = np.zeros((cfg.B, cfg.Hkv, Lmax, cfg.d), dtype=k.dtype)
    v2 = np.zeros_like(k2)
    for b in range(cfg.B):
        L0 = int(wl.lens[b])
        k2[b, :, :L0] = k[b, :, :L0]
        v2[b, :, :L0] = v[b, :, :L0]
        for s in range(nsteps):
            k2[b, :, L0 + s] = toks[s][0][b, :, 0]
            v2[b, :, L0 + s] = toks[s][1][b, :, 0]
    Dk, Uk, Dv, Uv = wl.proj_host
    return oracle.decode(qs[nsteps - 1], k2, v2, lens, Dk, Uk, Dv, Uv, cfg.w, cfg.dtype)


CFG = I.Decode("step", 130, 6, 8, 2, 64, 16, 96, "bf16", L_range=(90, 700), shuffle_pages=True)


def test_decode_step_equals_append_then_decode():
    """The fused step gives bit-identical cache bytes and outputs to the two
    calls made in turn, and matches the oracle."""
    nsteps = 5
    toks, qs = _steps(CFG, nsteps)
    a = W.DecodeWorkload(CFG, extra_tokens=nsteps, keep_history=True)
    b = W.DecodeWorkload(CFG, extra_tokens=nsteps)
    for s in range(nsteps):
        kn, vn = (W.upload(x, "bf16") for x in toks[s])
        q = W.upload(qs[s], "bf16")
        oa = dar.dar_decode_step(a.cache, kn, vn, a.Dk, a.Dv, q, a.Uk, a.Uv, a.workspace)
        dar.dar_cache_append(b.cache, kn, vn, b.Dk, b.Dv)
        ob = dar.dar_attn_decode(b.cache, q, b.Uk, b.Uv, b.workspace)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(W.download(oa), W.download(ob))
    for name in ("win_k", "win_v", "pool_kd", "pool_vd", "seq_lens"):
        np.testing.assert_array_equal(W.download(getattr(a.cache, name)), W.download(getattr(b.cache, name)))
    want = _oracle_after(a, toks, qs, nsteps)
    got = W.to_f64(W.download(oa), "bf16")
    assert np.abs(got - want).max() <= TOL
    assert a.cache.device_status() == 0


def test_decode_step_graph_matches_oracle():
    """Steps captured in one CUDA graph (the launch edges the benchmark
    replays, programmatic ones included) give the oracle's result."""
    nsteps = 4
    toks, qs = _steps(CFG, nsteps)
    wl = W.DecodeWorkload(CFG, extra_tokens=nsteps, keep_history=True)
    kn = [tuple(W.upload(x, "bf16") for x in toks[s]) for s in range(nsteps)]
    q = [W.upload(qs[s], "bf16") for s in range(nsteps)]
    out = torch.empty_like(wl.q)
    # the state a replay starts from: lengths and ring (the steps overwrite
    # ring slots that later migrations would otherwise read)
    saved = [t.clone() for t in (wl.cache.seq_lens, wl.cache.win_k, wl.cache.win_v)]
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for s in range(nsteps):
            dar.dar_decode_step(wl.cache, kn[s][0], kn[s][1], wl.Dk, wl.Dv, q[s], wl.Uk, wl.Uv, wl.workspace,
                                out=out)
    for _ in range(2):  # each replay starts from the restored state and recomputes the same steps
        for dst, src in zip((wl.cache.seq_lens, wl.cache.win_k, wl.cache.win_v), saved):
            dst.copy_(src)
        g.replay()
        torch.cuda.synchronize()
        got = W.to_f64(W.download(out), "bf16")
        want = _oracle_after(wl, toks, qs, nsteps)
        assert np.abs(got - want).max() <= TOL
    assert wl.cache.device_status() == 0


def test_decode_step_rejects_before_launching():
    """A bad decode argument refuses the whole step: the append does not run."""
    wl = W.DecodeWorkload(CFG, extra_tokens=1)
    kn, vn = (W.upload(x, "bf16") for x in I.decode_new_tokens(CFG, 0))
    lens = W.download(wl.cache.seq_lens).copy()
    small = torch.empty(16, dtype=torch.uint8, device="cuda")
    with pytest.raises(dar.DarError) as e:
        dar.dar_decode_step(wl.cache, kn, vn, wl.Dk, wl.Dv, wl.q, wl.Uk, wl.Uv, small)
    assert e.value.code == dar.DAR_ERR_CAPACITY
    torch.cuda.synchronize()
    np.testing.assert_array_equal(W.download(wl.cache.seq_lens), lens)
