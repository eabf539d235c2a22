"""GPU prefill parity against the CPU oracle (through the C ABI).

Tolerances: max-abs 1e-5 for fp32 storage, 2e-2 for bf16 storage (fp32
accumulation), comparing the kernel's output with the oracle's fp64 result.
"""
import numpy as np
import pytest

import oracle
from paper_2606_18587_gb300 import inputs as I

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("no CUDA device", allow_module_level=True)

from paper_2606_18587_gb300 import workloads as W  # noqa: E402

TOL = {"f32": 1e-5, "bf16": 2e-2}


def gpu_prefill(cfg):
    wl = W.PrefillWorkload(cfg)
    wl.run()
    torch.cuda.synchronize()
    return wl, W.to_f64(W.download(wl.out), cfg.dtype)


def oracle_prefill(wl, rows=None):
    x, cfg = wl.host, wl.cfg
    return oracle.prefill(x["q"], x["k"], x["v"], x["Dk"], x["Uk"], x["Dv"], x["Uv"], cfg.w, cfg.dtype, rows=rows)


def test_prefill_tiny_f32_full():
    """B1 H4 N256 d64 dd16 w32, fp32: every output element."""
    cfg = I.PREFILL_TINY_F32
    wl, got = gpu_prefill(cfg)
    want = oracle_prefill(wl)
    err = np.abs(got - want).max()
    assert err <= TOL["f32"], err


CASES = [
    # dtype, B, Hq, Hkv, N, dd, w
    ("f32", 1, 2, 2, 1, 16, 1),       # single token
    ("f32", 2, 4, 2, 130, 8, 0),      # w = 0: uniform reduction, ragged tail
    ("f32", 1, 2, 1, 97, 32, 200),    # window covers everything: plain causal attention
    ("f32", 1, 3, 3, 191, 64, 64),    # d_down = d
    ("bf16", 1, 4, 2, 200, 16, 37),   # GQA, band tiles with odd window
    ("bf16", 2, 2, 2, 257, 8, 1),     # only the current token is local
    ("bf16", 1, 8, 2, 320, 32, 128),  # G = 4
    ("bf16", 1, 2, 2, 64, 64, 63),
    ("bf16", 1, 2, 2, 700, 16, 512),  # the 410M-like window on a short sequence
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "-".join(map(str, c)))
def test_prefill_small_cases(case):
    dtype, B, Hq, Hkv, N, dd, w = case
    cfg = I.Prefill("case", 40 + N + dd + w, B, Hq, Hkv, N, 64, dd, w, dtype)
    wl, got = gpu_prefill(cfg)
    want = oracle_prefill(wl)
    err = np.abs(got - want).max()
    assert err <= TOL[dtype], err
    assert np.isfinite(got).all()


def test_prefill_410m_full_head_and_tile_edges():
    """B8 H16 N8192 d64 dd16 w512 bf16 at full size, in the configuration the
    benchmark times.  The oracle evaluates every row of one (b, h), and in all
    128 (b, h) the rows at tile and window edges (first, 63/64, 127/128, w - 1,
    w, w + 63, the last tiles, the last row) plus random rows."""
    cfg = I.PREFILL_410M
    wl, got = gpu_prefill(cfg)
    assert np.isfinite(got).all()
    rng = np.random.default_rng(0)
    N, w = cfg.N, cfg.w
    edges = [0, 1, 63, 64, 127, 128, w - 1, w, w + 1, w + 63, w + 64, N - 129, N - 128, N - 65, N - 64, N - 1]
    rows = [(5, 11, i) for i in range(N)]
    for b in range(cfg.B):
        for h in range(cfg.Hq):
            rows += [(b, h, i) for i in edges + list(rng.integers(0, N, 2))]
    rows = np.array(rows)
    want = oracle_prefill(wl, rows=rows)
    err = np.abs(got[rows[:, 0], rows[:, 1], rows[:, 2]] - want).max()
    assert err <= TOL["bf16"], err
