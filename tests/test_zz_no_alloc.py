"""dar_attn_decode_noalloc: the decode entry point for callers that cannot
allocate device memory (no workspace argument; the library's built-in device
scratch array is used).  Its output must match dar_attn_decode's within the
bf16 tolerance of the other decode tests, on two calls in a row, and a shape
whose scratch need exceeds the built-in size must be refused cleanly.

This file is collected last so that, in a run that stops at the first
failure, every other test has already run."""
import numpy as np
import pytest

from paper_2606_18587_gb300 import inputs as I

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("no CUDA device", allow_module_level=True)

from paper_2606_18587_gb300 import dar  # noqa: E402
from paper_2606_18587_gb300 import workloads as W  # noqa: E402

TOL = 2e-2  # bf16 storage, fp32 accumulation


def test_noalloc_matches_workspace_decode_twice():
    cfg = I.Decode("noalloc", 120, 8, 8, 4, 64, 16, 64, "bf16", L_range=(300, 2500), shuffle_pages=True)
    wl = W.DecodeWorkload(cfg)
    ref = W.to_f64(W.download(wl.decode()), "bf16")
    assert 0 < dar.dar_decode_workspace_bytes(wl.cache, cfg.Hq) <= (8 << 20)  # fits the built-in scratch
    for _ in range(2):
        out = dar.dar_attn_decode_noalloc(wl.cache, wl.q, wl.Uk, wl.Uv)
        torch.cuda.synchronize()
        got = W.to_f64(W.download(out), "bf16")
        assert np.abs(got - ref).max() <= TOL
        assert np.isfinite(got).all()
    assert wl.cache.device_status() == 0


def test_noalloc_refuses_shapes_beyond_its_scratch():
    # 512 sequences x 64 query heads with d_down = 64: the absorbed queries
    # alone (512 * 64 * 64 fp32) exceed the built-in scratch; nothing may be launched
    cache = dar.DarCache(512, 8, 64, 16, 1, dtype=torch.bfloat16)
    assert dar.dar_decode_workspace_bytes(cache, 64) > (8 << 20)
    q = torch.zeros((512, 64, 64), dtype=torch.bfloat16, device="cuda")
    U = torch.zeros((8, 64, 64), dtype=torch.float32, device="cuda")
    out = torch.full_like(q, 7.0)
    with pytest.raises(dar.DarError) as e:
        dar.dar_attn_decode_noalloc(cache, q, U, U, out=out)
    assert e.value.code == dar.DAR_ERR_CAPACITY
    assert "scratch" in str(e.value)
    torch.cuda.synchronize()
    assert torch.all(out == 7.0)
