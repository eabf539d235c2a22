"""The give-up path of the library's bounded waits, exercised on the GPU
without a fault: a kernel waits, with a short limit, on a barrier that
nothing completes.  The call must come back, the status word must read
DAR_ERR_DEVICE, and the next ordinary call must still be correct."""
import time

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


def test_starved_wait_reports_device_error_and_context_survives():
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    dar.dar_check_bounded_wait(status, 5000)  # 5 ms limit
    torch.cuda.synchronize()
    elapsed = time.perf_counter() - t0
    assert int(status.item()) == dar.DAR_ERR_DEVICE
    assert elapsed >= 0.004  # it really waited for its limit before giving up
    # the first error wins: a second give-up leaves the word as it is
    dar.dar_check_bounded_wait(status, 1000)
    torch.cuda.synchronize()
    assert int(status.item()) == dar.DAR_ERR_DEVICE
    # the device is still usable: an ordinary decode is correct
    cfg = I.Decode("after-giveup", 131, 3, 4, 2, 64, 16, 32, "bf16", L_range=(40, 300), shuffle_pages=True)
    wl = W.DecodeWorkload(cfg, keep_history=True)
    out = wl.decode()
    torch.cuda.synchronize()
    k, v = wl.history_arrays()
    Dk, Uk, Dv, Uv = wl.proj_host
    want = oracle.decode(wl.q_host, k, v, wl.lens, Dk, Uk, Dv, Uv, cfg.w, "bf16")
    assert np.abs(W.to_f64(W.download(out), "bf16") - want).max() <= 2e-2
    assert wl.cache.device_status() == 0
