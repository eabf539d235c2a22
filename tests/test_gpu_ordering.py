"""Ordering on the stream: dar_attn_decode reads q and Uk only once the work
ahead of it on the stream has finished, even when that work lets dependent
kernels start early (programmatic dependent launch).  A helper kernel triggers
its dependents at entry and writes the query only after a delay; the decode
must still see the written query.  dar_decode_step is checked the same way."""
import ctypes
import os
import shutil
import subprocess

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

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.fixture(scope="module")
def late_copy(tmp_path_factory):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    out = str(tmp_path_factory.mktemp("helpers") / "liblate_writer.so")
    subprocess.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O2", "-shared", "-Xcompiler", "-fPIC",
                    "-o", out, os.path.join(HERE, "helpers", "late_writer.cu")], check=True)
    lib = ctypes.CDLL(out)
    lib.late_copy.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int, ctypes.c_ulonglong, ctypes.c_void_p]
    lib.late_copy.restype = ctypes.c_int

    def run(src, dst, delay_ns=200_000):
        assert src.numel() * src.element_size() % 16 == 0
        rc = lib.late_copy(ctypes.c_void_p(src.data_ptr()), ctypes.c_void_p(dst.data_ptr()),
                           src.numel() * src.element_size() // 16, delay_ns,
                           ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
        assert rc == 0
    return run


CFG = I.Decode("ordering", 140, 4, 8, 2, 64, 16, 64, "bf16", L_range=(200, 900), shuffle_pages=True)


def _oracle(wl, q_host, extra=None):
    k, v = wl.history_arrays()
    lens = wl.lens.copy()
    if extra is not None:  # one appended token per sequence
        kn, vn = extra
        L = int(lens.max()) + 1
        k2 = np.zeros((CFG.B, CFG.Hkv, L, CFG.d), dtype=k.dtype)
        v2 = np.zeros_like(k2)
        for b in range(CFG.B):
            Lb = int(lens[b])
            k2[b, :, :Lb], v2[b, :, :Lb] = k[b, :, :Lb], v[b, :, :Lb]
            k2[b, :, Lb], v2[b, :, Lb] = kn[b, :, 0], vn[b, :, 0]
        k, v, lens = k2, v2, lens + 1
    Dk, Uk, Dv, Uv = wl.proj_host
    return oracle.decode(q_host, k, v, lens, Dk, Uk, Dv, Uv, CFG.w, CFG.dtype)


def test_decode_waits_for_a_writer_that_triggers_early(late_copy):
    wl = W.DecodeWorkload(CFG, keep_history=True)
    q_new_host = I.decode_query(CFG, step=7)
    q_src = W.upload(q_new_host, "bf16")
    q_dst = torch.zeros_like(q_src)  # stale until the helper's delayed copy
    torch.cuda.synchronize()
    late_copy(q_src, q_dst)
    out = dar.dar_attn_decode(wl.cache, q_dst, wl.Uk, wl.Uv, wl.workspace)
    torch.cuda.synchronize()
    got = W.to_f64(W.download(out), "bf16")
    assert np.abs(got - _oracle(wl, q_new_host)).max() <= 2e-2


def test_decode_step_waits_for_a_writer_that_triggers_early(late_copy):
    wl = W.DecodeWorkload(CFG, extra_tokens=1, keep_history=True)
    q_new_host = I.decode_query(CFG, step=8)
    kn_host, vn_host = I.decode_new_tokens(CFG, 3)
    q_src = W.upload(q_new_host, "bf16")
    q_dst = torch.zeros_like(q_src)
    kn, vn = W.upload(kn_host, "bf16"), W.upload(vn_host, "bf16")
    torch.cuda.synchronize()
    late_copy(q_src, q_dst)
    out = dar.dar_decode_step(wl.cache, kn, vn, wl.Dk, wl.Dv, q_dst, wl.Uk, wl.Uv, wl.workspace)
    torch.cuda.synchronize()
    got = W.to_f64(W.download(out), "bf16")
    assert np.abs(got - _oracle(wl, q_new_host, (kn_host, vn_host))).max() <= 2e-2
    assert wl.cache.device_status() == 0
