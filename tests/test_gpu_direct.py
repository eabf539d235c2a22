"""GPU parity of the direct lower-dimensional global attention (Sec. 5,
"Direct lower-dimensional global attention") against the CPU oracle, through
the C ABI: dar_attn_prefill_direct and dar_attn_decode_direct.  The global
path scores the row's own d_down query q^D against the cached k^D at
scale 1/sqrt(d_down) and maps the weighted v^D to d with Wo; the local path and
the one softmax are those of Eq. 3-4.  Tolerances as for the standard method:
max-abs 1e-5 (fp32 storage), 2e-2 (bf16 storage, fp32 accumulation)."""
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


def run_prefill(cfg):
    wl = W.PrefillWorkload(cfg)
    qd_host = I.direct_queries(cfg)
    qd = W.upload(qd_host, cfg.dtype)
    out = dar.dar_attn_prefill_direct(wl.q, qd, wl.k, wl.v, wl.Dk, wl.Dv, wl.Uv, cfg.w, workspace=wl.workspace)
    torch.cuda.synchronize()
    return wl, qd_host, W.to_f64(W.download(out), cfg.dtype)


def oracle_prefill(wl, qd_host, rows=None):
    x, cfg = wl.host, wl.cfg
    return oracle.prefill_direct(x["q"], qd_host, x["k"], x["v"], x["Dk"], x["Dv"], x["Uv"], cfg.w, cfg.dtype,
                                 rows=rows)


def test_prefill_direct_tiny_f32_full():
    """B1 H4 N256 d64 dd16 w32, fp32: every output element."""
    wl, qd, got = run_prefill(I.PREFILL_TINY_F32)
    err = np.abs(got - oracle_prefill(wl, qd)).max()
    assert err <= TOL["f32"], err


CASES = [
    # dtype, B, Hq, Hkv, N, dd, w
    ("f32", 2, 4, 2, 130, 8, 0),      # w = 0: every pair global, ragged tail
    ("f32", 1, 2, 1, 97, 32, 200),    # window covers everything: the global path plays no part
    ("f32", 1, 3, 3, 191, 64, 64),
    ("bf16", 1, 4, 2, 200, 16, 37),   # GQA, band tiles with odd window
    ("bf16", 2, 2, 2, 257, 8, 1),     # d_down = 8 (scale ratio sqrt(8)), only the current token local
    ("bf16", 1, 8, 2, 320, 32, 128),  # G = 4
    ("bf16", 1, 2, 2, 300, 64, 0),    # w = 0 with d_down = d
    ("bf16", 1, 2, 2, 700, 16, 512),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "-".join(map(str, c)))
def test_prefill_direct_small_cases(case):
    dtype, B, Hq, Hkv, N, dd, w = case
    cfg = I.Prefill("direct case", 70 + N + dd + w, B, Hq, Hkv, N, 64, dd, w, dtype)
    wl, qd, got = run_prefill(cfg)
    assert np.isfinite(got).all()
    err = np.abs(got - oracle_prefill(wl, qd)).max()
    assert err <= TOL[dtype], err


def test_prefill_direct_410m_shape_sampled():
    """B8 H16 N8192 d64 dd16 w512 bf16 at full size: every (b, h) at the tile
    and window edges plus random rows."""
    cfg = I.PREFILL_410M
    wl, qd, got = run_prefill(cfg)
    assert np.isfinite(got).all()
    rng = np.random.default_rng(3)
    N, w = cfg.N, cfg.w
    edges = [0, 63, 64, 127, 128, w - 1, w, w + 64, N - 129, N - 128, N - 1]
    rows = np.array([(b, h, i) for b in range(cfg.B) for h in range(cfg.Hq)
                     for i in edges + list(rng.integers(0, N, 2))])
    want = oracle_prefill(wl, qd, rows=rows)
    err = np.abs(got[rows[:, 0], rows[:, 1], rows[:, 2]] - want).max()
    assert err <= TOL["bf16"], err


def run_decode(cfg, heads=None):
    wl = W.DecodeWorkload(cfg, keep_history=True)
    qd_host = I.direct_queries(cfg)
    qd = W.upload(qd_host, cfg.dtype)
    out = dar.dar_attn_decode_direct(wl.cache, wl.q, qd, wl.Uv, wl.workspace)
    torch.cuda.synchronize()
    assert wl.cache.device_status() == 0
    got = W.to_f64(W.download(out), cfg.dtype)
    k, v = wl.history_arrays()
    Dk, _, Dv, Wo = wl.proj_host
    want = oracle.decode_direct(wl.q_host, qd_host, k, v, wl.lens, Dk, Dv, Wo, cfg.w, cfg.dtype, heads=heads)
    if heads is None:
        heads = [(b, h) for b in range(cfg.B) for h in range(cfg.Hq)]
    return max(np.abs(got[b, h] - want[b, h]).max() for b, h in heads), got


def test_decode_direct_160m_all_heads():
    """B32 H12 L4096 d64 dd16 w128 bf16: every (b, h)."""
    err, got = run_decode(I.DECODE_160M)
    assert np.isfinite(got).all()
    assert err <= TOL["bf16"], err


def test_decode_direct_1b_gqa_paged():
    """B64 Hq32 Hkv8 dd16 w256, ragged lengths, shuffled pages: one head of every
    sequence and every head of three sequences."""
    cfg = I.DECODE_1B_GQA
    heads = sorted({(b, h) for b in (0, 17, 42) for h in range(cfg.Hq)} | {(b, (7 * b) % cfg.Hq)
                                                                          for b in range(cfg.B)})
    err, got = run_decode(cfg, heads=heads)
    assert np.isfinite(got).all()
    assert err <= TOL["bf16"], err


@pytest.mark.parametrize("k", [0, 3, 5, 12])
def test_decode_direct_sweep_points(k):
    """Sweep points w64 dd8, w64 dd64, w256 dd16, w16384 dd8 (B16 H16 L16384):
    one head of every sequence."""
    cfg = I.sweep_point(k)
    heads = [(b, (5 * b + k) % cfg.Hq) for b in range(cfg.B)]
    err, _ = run_decode(cfg, heads=heads)
    assert err <= TOL["bf16"], err


def test_decode_direct_small_f32():
    """fp32 cache, ragged lengths around the window, GQA: every (b, h)."""
    cfg = I.Decode("direct decode f32 B5 Hq4 Hkv2 w40 dd8", 77, 5, 4, 2, 64, 8, 40, "f32", L_range=(1, 300),
                   shuffle_pages=True)
    err, _ = run_decode(cfg)
    assert err <= TOL["f32"], err
