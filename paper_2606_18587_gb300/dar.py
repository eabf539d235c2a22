"""Python binding of the DAR CUDA library (``include/dar.h``).

Argument marshalling only: every function passes device pointers, sizes and
the current CUDA stream straight to the C entry point of the same name; all
arithmetic runs in the sm_103a kernels.  PyTorch supplies device memory and
streams.  There is no fallback: if ``libdar_gb300.so`` is missing or a call
fails, an exception is raised.
"""
from __future__ import annotations

import ctypes
import os
import re

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libdar_gb300.so")
HEADER = os.path.join(os.path.dirname(_HERE), "include", "dar.h")

DAR_OK, DAR_ERR_INVALID_ARG, DAR_ERR_UNSUPPORTED, DAR_ERR_CAPACITY, DAR_ERR_CUDA, DAR_ERR_DEVICE = range(6)
DAR_F32, DAR_BF16 = 0, 1
PAGE_SIZE = 64
_TORCH_DTYPE = {DAR_F32: torch.float32, DAR_BF16: torch.bfloat16}
_CODE = {torch.float32: DAR_F32, torch.bfloat16: DAR_BF16}


class DarError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"DAR error {code}: {msg}")
        self.code = code


class dar_cache(ctypes.Structure):
    _fields_ = [
        ("dtype", ctypes.c_int),
        ("B", ctypes.c_int32), ("Hkv", ctypes.c_int32), ("d", ctypes.c_int32),
        ("d_down", ctypes.c_int32), ("w", ctypes.c_int32),
        ("max_pages_per_seq", ctypes.c_int32), ("num_pages", ctypes.c_int32),
        ("win_k", ctypes.c_void_p), ("win_v", ctypes.c_void_p),
        ("pool_kd", ctypes.c_void_p), ("pool_vd", ctypes.c_void_p),
        ("block_table", ctypes.c_void_p), ("seq_lens", ctypes.c_void_p), ("status", ctypes.c_void_p),
    ]


class dar_latent_cache(ctypes.Structure):
    _fields_ = [
        ("B", ctypes.c_int32), ("Hkv", ctypes.c_int32), ("d", ctypes.c_int32), ("D", ctypes.c_int32),
        ("d_lat", ctypes.c_int32), ("w", ctypes.c_int32),
        ("max_pages_per_seq", ctypes.c_int32), ("num_pages", ctypes.c_int32),
        ("win_k", ctypes.c_void_p), ("win_v", ctypes.c_void_p), ("pool_c", ctypes.c_void_p),
        ("block_table", ctypes.c_void_p), ("seq_lens", ctypes.c_void_p), ("status", ctypes.c_void_p),
    ]


_lib = None


def load_library(path: str = LIB_PATH):
    """Load the compiled library (raises if it was not built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"DAR CUDA library not found at {path}; build it with "
                           "`python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(path)
    P, I32, SZ, F = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t, ctypes.c_float
    LP = ctypes.POINTER(dar_latent_cache)
    CP = ctypes.POINTER(dar_cache)
    sig = {
        "dar_down_project": ([ctypes.c_int, I32, I32, I32, I32, I32, P, P, P, P], ctypes.c_int),
        "dar_cache_append": ([CP, P, P, I32, P, P, P, P], ctypes.c_int),
        "dar_decode_workspace_bytes": ([CP, I32], SZ),
        "dar_attn_decode": ([CP, I32, P, P, P, F, P, P, SZ, P], ctypes.c_int),
        "dar_attn_decode_noalloc": ([CP, I32, P, P, P, F, P, P], ctypes.c_int),
        "dar_decode_step": ([CP, P, P, I32, P, P, P, I32, P, P, P, F, P, P, SZ, P], ctypes.c_int),
        "dar_check_bounded_wait": ([P, ctypes.c_uint32, P], ctypes.c_int),
        "dar_prefill_workspace_bytes": ([ctypes.c_int, I32, I32, I32, I32], SZ),
        "dar_prefill_chunk_workspace_bytes": ([CP, I32], SZ),
        "dar_prefill_chunk": ([CP, I32, I32, P, P, P, P, P, P, P, F, P, P, SZ, P], ctypes.c_int),
        "dar_attn_prefill": ([ctypes.c_int, I32, I32, I32, I32, I32, I32, I32, P, P, P, P, P, P, P, F, P, P,
                              SZ, P, P], ctypes.c_int),
        "dar_attn_prefill_direct": ([ctypes.c_int, I32, I32, I32, I32, I32, I32, I32, P, P, P, P, P, P, P, F, F,
                                     P, P, SZ, P, P], ctypes.c_int),
        "dar_attn_decode_direct": ([CP, I32, P, P, P, F, F, P, P, SZ, P], ctypes.c_int),
        "dar_attn_backward_workspace_bytes": ([ctypes.c_int, I32, I32, I32, I32, I32], SZ),
        "dar_attn_backward": ([ctypes.c_int, I32, I32, I32, I32, I32, I32, I32] + [P] * 9 + [F] + [P] * 8 + [SZ, P],
                              ctypes.c_int),
        "dar_latent_append": ([LP, P, P, P, I32, P, P, P], ctypes.c_int),
        "dar_latent_absorb": ([I32, I32, I32, I32, P, P, P, P, P, P], ctypes.c_int),
        "dar_latent_decode_workspace_bytes": ([LP, I32], SZ),
        "dar_latent_decode": ([LP, I32, P, P, P, F, P, P, SZ, P], ctypes.c_int),
        "dar_last_error": ([], ctypes.c_char_p),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    _lib = lib
    return lib


def declared_symbols(header: str = HEADER):
    """Names of the functions include/dar.h declares."""
    text = open(header).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w\s\*]*?\b(dar_\w+)\s*\(", text, re.M)))


def dar_last_error() -> str:
    return load_library().dar_last_error().decode()


def _check(code):
    if code != DAR_OK:
        raise DarError(code, dar_last_error())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else ctypes.c_void_p(0)


def _dev(t, name, dtype=None):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    return t


def _code(t):
    if t.dtype not in _CODE:
        raise ValueError(f"unsupported dtype {t.dtype}")
    return _CODE[t.dtype]


# --------------------------------------------------------------------------- Eq. 1

def dar_down_project(x, W, out=None, stream=None):
    """Eq. 1 per KV head: ``x [B,Hkv,n,d]`` (T) times ``W [Hkv,d,dd]`` (fp32) -> ``[B,Hkv,n,dd]`` (T)."""
    _dev(x, "x")
    _dev(W, "W", torch.float32)
    B, Hkv, n, d = x.shape
    dd = W.shape[2]
    if out is None:
        out = torch.empty((B, Hkv, n, dd), dtype=x.dtype, device=x.device)
    _dev(out, "out", x.dtype)
    _check(load_library().dar_down_project(_code(x), B, Hkv, n, d, dd, _ptr(x), _ptr(W), _ptr(out),
                                           _stream(stream)))
    return out


# --------------------------------------------------------------------------- cache

class DarCache:
    """Caller-owned mixed-dimension cache (device tensors) and its ``dar_cache`` struct.

    ``block_table`` (int32 ``[B, max_pages_per_seq]``) maps each sequence's
    logical pages to physical pages of the pools; by default sequence b owns
    pages ``b*max_pages_per_seq ..`` in order."""

    def __init__(self, B, Hkv, d_down, w, max_pages_per_seq, num_pages=None, dtype=torch.bfloat16,
                 block_table=None, device="cuda", d=64):
        self.dtype = dtype
        self.B, self.Hkv, self.d, self.d_down, self.w = B, Hkv, d, d_down, w
        self.max_pages_per_seq = max_pages_per_seq
        if num_pages is None:
            num_pages = B * max_pages_per_seq
        self.num_pages = num_pages
        self.win_k = torch.zeros((B, Hkv, w, d), dtype=dtype, device=device)
        self.win_v = torch.zeros_like(self.win_k)
        self.pool_kd = torch.zeros((max(num_pages, 1), Hkv, PAGE_SIZE, d_down), dtype=dtype, device=device)
        self.pool_vd = torch.zeros_like(self.pool_kd)
        if block_table is None:
            block_table = torch.arange(B * max_pages_per_seq, dtype=torch.int32).reshape(B, max_pages_per_seq)
        self.block_table = torch.as_tensor(block_table, dtype=torch.int32).to(device).contiguous()
        if self.block_table.numel() == 0:
            self.block_table = torch.full((max(B, 1), 1), -1, dtype=torch.int32, device=device)
        self.seq_lens = torch.zeros(B, dtype=torch.int32, device=device)
        self.status = torch.zeros(1, dtype=torch.int32, device=device)
        self._struct = dar_cache(
            _CODE[dtype], B, Hkv, d, d_down, w, max_pages_per_seq, num_pages,
            self.win_k.data_ptr(), self.win_v.data_ptr(), self.pool_kd.data_ptr(), self.pool_vd.data_ptr(),
            self.block_table.data_ptr(), self.seq_lens.data_ptr(), self.status.data_ptr())

    @property
    def struct(self):
        return ctypes.byref(self._struct)

    def device_status(self) -> int:
        return int(self.status.item())


def dar_cache_append(cache: DarCache, k_new, v_new, Dk, Dv, n_per_seq=None, stream=None):
    """Append ``k_new, v_new [B,Hkv,n,d]`` (first ``n_per_seq[b]`` rows of sequence b)."""
    _dev(k_new, "k_new", cache.dtype)
    _dev(v_new, "v_new", cache.dtype)
    _dev(Dk, "Dk", torch.float32)
    _dev(Dv, "Dv", torch.float32)
    if n_per_seq is not None:
        _dev(n_per_seq, "n_per_seq", torch.int32)
    n = k_new.shape[2]
    _check(load_library().dar_cache_append(cache.struct, _ptr(k_new), _ptr(v_new), n, _ptr(n_per_seq),
                                           _ptr(Dk), _ptr(Dv), _stream(stream)))


def dar_decode_workspace_bytes(cache: DarCache, Hq: int) -> int:
    return int(load_library().dar_decode_workspace_bytes(cache.struct, Hq))


def decode_workspace(cache: DarCache, Hq: int):
    """A workspace of the size dar_attn_decode needs (no initialisation needed)."""
    nbytes = dar_decode_workspace_bytes(cache, Hq)
    if nbytes == 0:
        raise DarError(DAR_ERR_INVALID_ARG, dar_last_error() or "bad cache/Hq")
    return torch.empty(nbytes, dtype=torch.uint8, device=cache.win_k.device)


def dar_attn_decode(cache: DarCache, q, Uk, Uv, workspace, scale=0.0, out=None, stream=None):
    """One decode step for queries ``q [B,Hq,d]`` at the last position of each sequence."""
    _dev(q, "q", cache.dtype)
    _dev(Uk, "Uk", torch.float32)
    _dev(Uv, "Uv", torch.float32)
    _dev(workspace, "workspace")
    if out is None:
        out = torch.empty_like(q)
    _dev(out, "out", cache.dtype)
    Hq = q.shape[1]
    _check(load_library().dar_attn_decode(cache.struct, Hq, _ptr(q), _ptr(Uk), _ptr(Uv), float(scale),
                                          _ptr(out), _ptr(workspace), workspace.numel() * workspace.element_size(),
                                          _stream(stream)))
    return out


def dar_decode_step(cache: DarCache, k_new, v_new, Dk, Dv, q, Uk, Uv, workspace, scale=0.0, out=None,
                    n_per_seq=None, stream=None):
    """dar_cache_append of ``k_new, v_new [B,Hkv,n,d]`` then dar_attn_decode of
    ``q [B,Hq,d]``, in one call (the decode's query set-up overlaps the append)."""
    _dev(k_new, "k_new", cache.dtype)
    _dev(v_new, "v_new", cache.dtype)
    _dev(Dk, "Dk", torch.float32)
    _dev(Dv, "Dv", torch.float32)
    _dev(q, "q", cache.dtype)
    _dev(Uk, "Uk", torch.float32)
    _dev(Uv, "Uv", torch.float32)
    _dev(workspace, "workspace")
    if n_per_seq is not None:
        _dev(n_per_seq, "n_per_seq", torch.int32)
    if out is None:
        out = torch.empty_like(q)
    _dev(out, "out", cache.dtype)
    _check(load_library().dar_decode_step(
        cache.struct, _ptr(k_new), _ptr(v_new), k_new.shape[2], _ptr(n_per_seq), _ptr(Dk), _ptr(Dv), q.shape[1],
        _ptr(q), _ptr(Uk), _ptr(Uv), float(scale), _ptr(out), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))
    return out


def dar_check_bounded_wait(status, limit_us: int, stream=None):
    """Run the library's wait-gives-up path on a barrier nothing completes;
    ``status`` (device int32) receives DAR_ERR_DEVICE after ``limit_us``."""
    _dev(status, "status", torch.int32)
    _check(load_library().dar_check_bounded_wait(_ptr(status), int(limit_us), _stream(stream)))


def dar_attn_decode_noalloc(cache: DarCache, q, Uk, Uv, scale=0.0, out=None, stream=None):
    """dar_attn_decode without a caller workspace: the library's built-in device
    scratch array is used instead (for callers that cannot allocate).  Calls
    that overlap on the device share that array and must be serialised."""
    _dev(q, "q", cache.dtype)
    _dev(Uk, "Uk", torch.float32)
    _dev(Uv, "Uv", torch.float32)
    if out is None:
        out = torch.empty_like(q)
    _dev(out, "out", cache.dtype)
    _check(load_library().dar_attn_decode_noalloc(cache.struct, q.shape[1], _ptr(q), _ptr(Uk), _ptr(Uv),
                                                  float(scale), _ptr(out), _stream(stream)))
    return out


# --------------------------------------------------------------------------- prefill

def dar_prefill_workspace_bytes(dtype, B, Hkv, N, d_down) -> int:
    return int(load_library().dar_prefill_workspace_bytes(_CODE[dtype], B, Hkv, N, d_down))


def dar_attn_prefill(q, k, v, Dk, Uk, Dv, Uv, w, scale=0.0, out=None, workspace=None, status=None,
                     stream=None):
    """Causal forward: ``q [B,Hq,N,d]``, ``k, v [B,Hkv,N,d]`` -> ``[B,Hq,N,d]``.
    ``status`` is an optional device int32 tensor receiving device-side errors."""
    _dev(q, "q")
    _dev(k, "k", q.dtype)
    _dev(v, "v", q.dtype)
    for name, t in (("Dk", Dk), ("Uk", Uk), ("Dv", Dv), ("Uv", Uv)):
        _dev(t, name, torch.float32)
    B, Hq, N, d = q.shape
    Hkv = k.shape[1]
    dd = Dk.shape[2]
    if out is None:
        out = torch.empty_like(q)
    _dev(out, "out", q.dtype)
    if workspace is None:
        workspace = torch.empty(max(1, dar_prefill_workspace_bytes(q.dtype, B, Hkv, N, dd)),
                                dtype=torch.uint8, device=q.device)
    _dev(workspace, "workspace")
    if status is not None:
        _dev(status, "status", torch.int32)
    _check(load_library().dar_attn_prefill(
        _code(q), B, Hq, Hkv, N, d, dd, int(w), _ptr(q), _ptr(k), _ptr(v), _ptr(Dk), _ptr(Uk), _ptr(Dv), _ptr(Uv),
        float(scale), _ptr(out), _ptr(workspace), workspace.numel(), _ptr(status), _stream(stream)))
    return out


def dar_attn_prefill_direct(q, qd, k, v, Dk, Dv, Wo, w, scale=0.0, scale_down=0.0, out=None, workspace=None,
                            status=None, stream=None):
    """Causal forward with the direct lower-dimensional global path (Sec. 5):
    ``qd [B,Hq,N,d_down]`` the global path's queries, ``Wo [Hkv,d_down,d]`` its
    output map; otherwise as :func:`dar_attn_prefill`."""
    _dev(q, "q")
    _dev(qd, "qd", q.dtype)
    _dev(k, "k", q.dtype)
    _dev(v, "v", q.dtype)
    for name, t in (("Dk", Dk), ("Dv", Dv), ("Wo", Wo)):
        _dev(t, name, torch.float32)
    B, Hq, N, d = q.shape
    Hkv = k.shape[1]
    dd = Dk.shape[2]
    if tuple(qd.shape) != (B, Hq, N, dd):
        raise ValueError(f"qd has shape {tuple(qd.shape)}, expected {(B, Hq, N, dd)}")
    if out is None:
        out = torch.empty_like(q)
    _dev(out, "out", q.dtype)
    if workspace is None:
        workspace = torch.empty(max(1, dar_prefill_workspace_bytes(q.dtype, B, Hkv, N, dd)),
                                dtype=torch.uint8, device=q.device)
    _dev(workspace, "workspace")
    if status is not None:
        _dev(status, "status", torch.int32)
    _check(load_library().dar_attn_prefill_direct(
        _code(q), B, Hq, Hkv, N, d, dd, int(w), _ptr(q), _ptr(qd), _ptr(k), _ptr(v), _ptr(Dk), _ptr(Dv), _ptr(Wo),
        float(scale), float(scale_down), _ptr(out), _ptr(workspace), workspace.numel(), _ptr(status),
        _stream(stream)))
    return out


def dar_attn_decode_direct(cache: DarCache, q, qd, Wo, workspace, scale=0.0, scale_down=0.0, out=None,
                           stream=None):
    """One decode step with the direct lower-dimensional global path (Sec. 5):
    ``qd [B,Hq,d_down]`` the global path's queries, ``Wo [Hkv,d_down,d]`` its
    output map; otherwise as :func:`dar_attn_decode`."""
    _dev(q, "q", cache.dtype)
    _dev(qd, "qd", cache.dtype)
    _dev(Wo, "Wo", torch.float32)
    _dev(workspace, "workspace")
    if tuple(qd.shape) != (q.shape[0], q.shape[1], cache.d_down):
        raise ValueError(f"qd has shape {tuple(qd.shape)}, expected {(q.shape[0], q.shape[1], cache.d_down)}")
    if out is None:
        out = torch.empty_like(q)
    _dev(out, "out", cache.dtype)
    _check(load_library().dar_attn_decode_direct(
        cache.struct, q.shape[1], _ptr(q), _ptr(qd), _ptr(Wo), float(scale), float(scale_down), _ptr(out),
        _ptr(workspace), workspace.numel() * workspace.element_size(), _stream(stream)))
    return out


def dar_attn_backward_workspace_bytes(dtype, B, Hq, Hkv, N, d_down) -> int:
    return int(load_library().dar_attn_backward_workspace_bytes(_CODE[dtype], B, Hq, Hkv, N, d_down))


def dar_attn_backward(q, k, v, Dk, Uk, Dv, Uv, out, dout, w, scale=0.0, workspace=None, grads=None,
                      stream=None):
    """Gradients of the causal forward (Sec. 2.3 training) for the output
    gradient ``dout``; ``out`` is the forward's output.  Returns a dict with
    ``dq, dk, dv`` (storage type) and ``dDk, dUk, dDv, dUv`` (fp32); ``grads``
    may hold preallocated tensors under those names."""
    _dev(q, "q")
    for name, t in (("k", k), ("v", v), ("out", out), ("dout", dout)):
        _dev(t, name, q.dtype)
    for name, t in (("Dk", Dk), ("Uk", Uk), ("Dv", Dv), ("Uv", Uv)):
        _dev(t, name, torch.float32)
    B, Hq, N, d = q.shape
    Hkv = k.shape[1]
    dd = Dk.shape[2]
    g = dict(grads or {})
    for name, like in (("dq", q), ("dk", k), ("dv", v), ("dDk", Dk), ("dUk", Uk), ("dDv", Dv), ("dUv", Uv)):
        if name not in g:
            g[name] = torch.empty_like(like)
        _dev(g[name], name, like.dtype)
    if workspace is None:
        workspace = torch.empty(max(1, dar_attn_backward_workspace_bytes(q.dtype, B, Hq, Hkv, N, dd)),
                                dtype=torch.uint8, device=q.device)
    _dev(workspace, "workspace")
    _check(load_library().dar_attn_backward(
        _code(q), B, Hq, Hkv, N, d, dd, int(w), _ptr(q), _ptr(k), _ptr(v), _ptr(Dk), _ptr(Uk), _ptr(Dv), _ptr(Uv),
        _ptr(out), _ptr(dout), float(scale), *(_ptr(g[n]) for n in ("dq", "dk", "dv", "dDk", "dUk", "dDv", "dUv")),
        _ptr(workspace), workspace.numel(), _stream(stream)))
    return g


def dar_prefill_chunk_workspace_bytes(cache: DarCache, n: int) -> int:
    return int(load_library().dar_prefill_chunk_workspace_bytes(cache.struct, int(n)))


def dar_prefill_chunk(cache: DarCache, q, k_new, v_new, Dk, Uk, Dv, Uv, scale=0.0, out=None, workspace=None,
                      stream=None):
    """Chunked prefill over the cache: queries ``q [B,Hq,n,d]`` at positions
    ``seq_lens[b] ..`` attend to the cache and causally within the chunk;
    ``k_new, v_new [B,Hkv,n,d]`` are then appended.  Returns ``[B,Hq,n,d]``."""
    _dev(q, "q", cache.dtype)
    _dev(k_new, "k_new", cache.dtype)
    _dev(v_new, "v_new", cache.dtype)
    for name, t in (("Dk", Dk), ("Uk", Uk), ("Dv", Dv), ("Uv", Uv)):
        _dev(t, name, torch.float32)
    B, Hq, n, d = q.shape
    if out is None:
        out = torch.empty_like(q)
    _dev(out, "out", cache.dtype)
    if workspace is None:
        workspace = torch.empty(max(1, dar_prefill_chunk_workspace_bytes(cache, n)), dtype=torch.uint8,
                                device=q.device)
    _dev(workspace, "workspace")
    _check(load_library().dar_prefill_chunk(
        cache.struct, Hq, n, _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(Dk), _ptr(Uk), _ptr(Dv), _ptr(Uv),
        float(scale), _ptr(out), _ptr(workspace), workspace.numel() * workspace.element_size(), _stream(stream)))
    return out


# --------------------------------------------------------------------------- latent form

class DarLatentCache:
    """Caller-owned cache of the latent form (one bottleneck per token shared
    by all heads, keys and values; full keys/values for the last ``w``
    tokens), and its ``dar_latent_cache`` struct.  bf16."""

    def __init__(self, B, Hkv, D, d_lat, w, max_pages_per_seq, num_pages=None, block_table=None, device="cuda",
                 d=64):
        self.B, self.Hkv, self.d, self.D, self.d_lat, self.w = B, Hkv, d, D, d_lat, w
        self.dtype = torch.bfloat16
        self.max_pages_per_seq = max_pages_per_seq
        if num_pages is None:
            num_pages = B * max_pages_per_seq
        self.num_pages = num_pages
        self.win_k = torch.zeros((B, Hkv, w, d), dtype=torch.bfloat16, device=device)
        self.win_v = torch.zeros_like(self.win_k)
        self.pool_c = torch.zeros((max(num_pages, 1), PAGE_SIZE, d_lat), dtype=torch.bfloat16, device=device)
        if block_table is None:
            block_table = torch.arange(B * max_pages_per_seq, dtype=torch.int32).reshape(B, max_pages_per_seq)
        self.block_table = torch.as_tensor(block_table, dtype=torch.int32).to(device).contiguous()
        self.seq_lens = torch.zeros(B, dtype=torch.int32, device=device)
        self.status = torch.zeros(1, dtype=torch.int32, device=device)
        self._struct = dar_latent_cache(
            B, Hkv, d, D, d_lat, w, max_pages_per_seq, num_pages, self.win_k.data_ptr(), self.win_v.data_ptr(),
            self.pool_c.data_ptr(), self.block_table.data_ptr(), self.seq_lens.data_ptr(), self.status.data_ptr())

    @property
    def struct(self):
        return ctypes.byref(self._struct)

    def device_status(self) -> int:
        return int(self.status.item())


def dar_latent_append(cache: DarLatentCache, h_new, k_new, v_new, W_down, n_per_seq=None, stream=None):
    """Append tokens: hidden states ``h_new [B,n,D]`` (their bottleneck c = h W_down
    is computed and cached), keys/values ``k_new, v_new [B,Hkv,n,d]``."""
    _dev(h_new, "h_new", torch.bfloat16)
    _dev(k_new, "k_new", torch.bfloat16)
    _dev(v_new, "v_new", torch.bfloat16)
    _dev(W_down, "W_down", torch.float32)
    if n_per_seq is not None:
        _dev(n_per_seq, "n_per_seq", torch.int32)
    _check(load_library().dar_latent_append(cache.struct, _ptr(h_new), _ptr(k_new), _ptr(v_new), k_new.shape[2],
                                            _ptr(n_per_seq), _ptr(W_down), _stream(stream)))


def dar_latent_absorb(W_up, W_K, W_V, stream=None):
    """``A_K = W_up W_K``, ``A_V = W_up W_V`` per KV head: ``W_up [d_lat,D]``,
    ``W_K, W_V [Hkv,D,d]`` -> ``A_K [Hkv,d,d_lat]`` (transposed) and ``A_V
    [Hkv,d_lat,d]``, fp32."""
    for name, t in (("W_up", W_up), ("W_K", W_K), ("W_V", W_V)):
        _dev(t, name, torch.float32)
    Hkv, D, d = W_K.shape
    d_lat = W_up.shape[0]
    A_K = torch.empty((Hkv, d, d_lat), dtype=torch.float32, device=W_up.device)
    A_V = torch.empty((Hkv, d_lat, d), dtype=torch.float32, device=W_up.device)
    _check(load_library().dar_latent_absorb(Hkv, D, d, d_lat, _ptr(W_up), _ptr(W_K), _ptr(W_V), _ptr(A_K),
                                            _ptr(A_V), _stream(stream)))
    return A_K, A_V


def latent_decode_workspace(cache: DarLatentCache, Hq: int):
    nbytes = int(load_library().dar_latent_decode_workspace_bytes(cache.struct, Hq))
    if nbytes == 0:
        raise DarError(DAR_ERR_INVALID_ARG, dar_last_error() or "bad latent cache/Hq")
    return torch.empty(nbytes, dtype=torch.uint8, device=cache.win_k.device)


def dar_latent_decode(cache: DarLatentCache, q, A_K, A_V, workspace, scale=0.0, out=None, stream=None):
    """One decode step of the latent form for ``q [B,Hq,d]`` (bf16)."""
    _dev(q, "q", torch.bfloat16)
    _dev(A_K, "A_K", torch.float32)
    _dev(A_V, "A_V", torch.float32)
    _dev(workspace, "workspace")
    if out is None:
        out = torch.empty_like(q)
    _dev(out, "out", torch.bfloat16)
    _check(load_library().dar_latent_decode(cache.struct, q.shape[1], _ptr(q), _ptr(A_K), _ptr(A_V), float(scale),
                                            _ptr(out), _ptr(workspace), workspace.numel(), _stream(stream)))
    return out
