"""GPU parity of the backward pass (dar_attn_backward, the training mode of
Sec. 2.3) against the CPU oracle's gradients (oracle.backward), through the
C ABI.

Each gradient tensor is compared element by element with the oracle's, with
max-abs error <= tol * max(1, max |oracle|): tol = 1e-5 for fp32 storage and
2e-2 for bf16 storage (fp32 accumulation; dq, dk, dv rounded to bf16).  The
scale factor lets the projection gradients, sums over every token of the
batch, be judged relative to their size.  The fp32 cases give the kernel the
oracle's forward output (rounded to fp32) so that they test the backward
alone; the bf16 cases give it the GPU forward's output, as training does."""
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
NAMES = ("dq", "dk", "dv", "dDk", "dUk", "dDv", "dUv")


def run_case(cfg):
    wl = W.PrefillWorkload(cfg)
    x = wl.host
    dout_host = I.normal_array(cfg.seed, I.S_QD, (cfg.B, cfg.Hq, cfg.N, cfg.d), dtype=cfg.dtype, sub=1)
    if cfg.dtype == "f32":
        o = oracle.prefill(x["q"], x["k"], x["v"], x["Dk"], x["Uk"], x["Dv"], x["Uv"], cfg.w, "f32")
        out = W.upload(o.astype(np.float32), "f32")
    else:
        wl.run()
        out = wl.out
    g = dar.dar_attn_backward(wl.q, wl.k, wl.v, wl.Dk, wl.Uk, wl.Dv, wl.Uv, out, W.upload(dout_host, cfg.dtype),
                              cfg.w)
    torch.cuda.synchronize()
    want = oracle.backward(x["q"], x["k"], x["v"], x["Dk"], x["Uk"], x["Dv"], x["Uv"], dout_host, cfg.w, cfg.dtype)
    errs = {}
    for n in NAMES:
        t = g[n]
        got = W.to_f64(W.download(t), cfg.dtype) if t.dtype != torch.float32 else t.cpu().numpy().astype(np.float64)
        assert np.isfinite(got).all(), n
        errs[n] = (float(np.abs(got - want[n]).max()), max(1.0, float(np.abs(want[n]).max())))
    return errs


def check(errs, dtype):
    bad = {n: e for n, e in errs.items() if not e[0] <= TOL[dtype] * e[1]}
    assert not bad, bad


CASES = [
    # dtype, B, Hq, Hkv, N, dd, w
    ("f32", 1, 4, 4, 256, 16, 32),     # the fp32 prefill workload's shape
    ("f32", 2, 4, 2, 130, 8, 0),       # w = 0: every pair global, GQA, ragged tail
    ("f32", 1, 2, 1, 97, 32, 200),     # window covers everything: projections get zero
    ("f32", 1, 3, 3, 191, 64, 64),
    ("bf16", 1, 4, 2, 200, 16, 37),
    ("bf16", 2, 2, 2, 257, 8, 1),
    ("bf16", 1, 8, 2, 320, 32, 128),   # G = 4
    ("bf16", 1, 2, 2, 700, 16, 512),
    ("bf16", 1, 2, 1, 1000, 64, 100),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "-".join(map(str, c)))
def test_backward_small_cases(case):
    dtype, B, Hq, Hkv, N, dd, w = case
    cfg = I.Prefill("backward case", 90 + N + dd + w, B, Hq, Hkv, N, 64, dd, w, dtype)
    check(run_case(cfg), dtype)


def test_backward_410m_sequence_length():
    """The 410M-like shape at its full sequence length (N8192 d64 dd16 w512
    bf16) on two heads: every gradient element."""
    p = I.PREFILL_410M
    cfg = I.Prefill("backward 410M-like B1 H2", p.seed, 1, 2, 2, p.N, p.d, p.dd, p.w, "bf16")
    check(run_case(cfg), "bf16")


def test_backward_repeat_is_bit_identical():
    """Every sum runs in a fixed order: two calls give the same bytes."""
    cfg = I.Prefill("backward determinism", 5, 2, 4, 2, 300, 64, 16, 50, "bf16")
    wl = W.PrefillWorkload(cfg)
    wl.run()
    dout = W.upload(I.normal_array(5, I.S_QD, (2, 4, 300, 64), dtype="bf16", sub=1), "bf16")
    a = dar.dar_attn_backward(wl.q, wl.k, wl.v, wl.Dk, wl.Uk, wl.Dv, wl.Uv, wl.out, dout, cfg.w)
    a = {n: t.clone() for n, t in a.items()}
    b = dar.dar_attn_backward(wl.q, wl.k, wl.v, wl.Dk, wl.Uk, wl.Dv, wl.Uv, wl.out, dout, cfg.w)
    for n in NAMES:
        assert torch.equal(a[n], b[n]), n
