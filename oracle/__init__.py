"""CPU oracle for DAR attention -- TEST INFRASTRUCTURE ONLY.

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product path (the CUDA library and
its Python binding) never calls it, and it shares no code with that path.

The arithmetic lives in ``dar_oracle.c`` (plain C, fp64 after the fp32
down-projection chain); this module compiles it with gcc and marshals numpy
arrays.  Function-level citations:

* :func:`down_project` -- Eq. 1 (bottleneck ``h^D = h W_down``), stored in the
  storage type with one fp32 FMA chain per element.
* :func:`attention_rows` -- Eq. 2 (explicit lift ``h' = h^D W_up``), Eq. 3
  (selection by ``i - j < w``) and Eq. 4 (one softmax over all ``j <= i``).
* :func:`prefill`, :func:`decode` -- the two row sets the method is used with:
  every position (training-mode forward), or the last position of each
  sequence (one inference step).
* :func:`backward` -- Sec. 2.3 (training): the gradients of the causal
  forward with respect to q, k, v and the four projections, by the chain rule
  through Eq. 4, 3, 2 and 1 in turn.
* :func:`latent_rows`, :func:`latent_prefill`, :func:`latent_decode` -- Eq. 1-4
  in the paper's own form on hidden states with one bottleneck per token
  shared by every head, keys and values (``c = h W_down``, ``h' = c W_up``,
  distant keys/values ``h' W_K``, ``h' W_V``), the cache scheme of Sec. 5.
* :func:`attention_rows_direct`, :func:`prefill_direct`, :func:`decode_direct`
  -- Sec. 5, "Direct lower-dimensional global attention": the global path in
  d_down with a query of its own and an output map of the global values.

Storage types: ``"f32"`` arrays are float32; ``"bf16"`` arrays are uint16
holding bfloat16 bit patterns.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dar_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_DTYPES = {"f32": 0, "bf16": 1}
_lib = None


def build(force: bool = False) -> str:
    """Compile ``dar_oracle.c`` into ``liboracle.so`` (gcc, no FMA contraction)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + ".%d.tmp" % os.getpid()
        subprocess.run(
            ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared",
             "-o", tmp, _SRC, "-lm", "-lpthread"],
            check=True,
        )
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        lib.dar_oracle_down_project.argtypes = [ctypes.c_int] * 6 + [P, P, P]
        lib.dar_oracle_down_project.restype = None
        lib.dar_oracle_f32_to_bf16.argtypes = [P, P, ctypes.c_size_t]
        lib.dar_oracle_f32_to_bf16.restype = None
        lib.dar_oracle_attention.argtypes = (
            [ctypes.c_int] * 8 + [P] * 7 + [ctypes.c_double, ctypes.c_long, P, P, P, P, ctypes.c_int]
        )
        lib.dar_oracle_attention.restype = ctypes.c_int
        lib.dar_oracle_attention_direct.argtypes = (
            [ctypes.c_int] * 8 + [P] * 7 + [ctypes.c_double, ctypes.c_double, ctypes.c_long, P, P, P, P, ctypes.c_int]
        )
        lib.dar_oracle_attention_direct.restype = ctypes.c_int
        lib.dar_oracle_backward.argtypes = (
            [ctypes.c_int] * 8 + [P] * 8 + [ctypes.c_double] + [P] * 7 + [ctypes.c_int]
        )
        lib.dar_oracle_backward.restype = ctypes.c_int
        lib.dar_oracle_attention_latent.argtypes = (
            [ctypes.c_int] * 9 + [P] * 7 + [ctypes.c_double, ctypes.c_long, P, P, P, P, ctypes.c_int]
        )
        lib.dar_oracle_attention_latent.restype = ctypes.c_int
        _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"], "oracle inputs must be C-contiguous"
    return ctypes.c_void_p(a.ctypes.data)


def _check(a: np.ndarray, dtype: str):
    want = np.float32 if dtype == "f32" else np.uint16
    if a.dtype != want:
        raise TypeError(f"expected {want} array for storage type {dtype}, got {a.dtype}")
    return np.ascontiguousarray(a)


def f32_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 bit patterns (nearest, ties to even)."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    _load().dar_oracle_f32_to_bf16(_ptr(x), _ptr(out), x.size)
    return out


def to_f64(a: np.ndarray, dtype: str) -> np.ndarray:
    """Exact conversion of a storage-type array to float64."""
    if dtype == "f32":
        return a.astype(np.float64)
    return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def down_project(x: np.ndarray, Dw: np.ndarray, dtype: str) -> np.ndarray:
    """Eq. 1 per KV head: ``x [B,Hkv,n,d]`` times ``Dw [Hkv,d,dd]`` -> ``[B,Hkv,n,dd]``.

    Each element is ``fmaf(x[t], Dw[t,c], acc)`` for t = 0..d-1 from +0.0f,
    rounded once to the storage type (round to nearest even)."""
    x = _check(x, dtype)
    Dw = np.ascontiguousarray(Dw, dtype=np.float32)
    B, Hkv, n, d = x.shape
    assert Dw.shape[0] == Hkv and Dw.shape[1] == d
    dd = Dw.shape[2]
    out = np.empty((B, Hkv, n, dd), dtype=x.dtype)
    _load().dar_oracle_down_project(_DTYPES[dtype], B, Hkv, n, d, dd, _ptr(x), _ptr(Dw), _ptr(out))
    return out


def attention_rows(q_rows, Hq, k, v, kd, vd, Uk, Uv, w, dtype, rows, scale=None, nthreads=None):
    """Eq. 2-4 for an explicit list of query rows.

    ``rows`` is an int array ``[R,3]`` of ``(b, h, i)``; ``q_rows [R,d]`` holds the
    query vector of each row, for a model with ``Hq`` query heads.  ``k, v
    [B,Hkv,N,d]`` and ``kd, vd [B,Hkv,N,dd]`` (Eq. 1 output) are in the storage
    type; ``Uk, Uv [Hkv,dd,d]`` are float32.  Returns float64 ``[R,d]``."""
    q_rows, k, v, kd, vd = (_check(a, dtype) for a in (q_rows, k, v, kd, vd))
    Uk = np.ascontiguousarray(Uk, dtype=np.float32)
    Uv = np.ascontiguousarray(Uv, dtype=np.float32)
    B, Hkv, N, d = k.shape
    dd = kd.shape[3]
    rows = np.ascontiguousarray(rows, dtype=np.int32).reshape(-1, 3)
    assert q_rows.shape == (rows.shape[0], d)
    rb = np.ascontiguousarray(rows[:, 0])
    rh = np.ascontiguousarray(rows[:, 1])
    ri = np.ascontiguousarray(rows[:, 2])
    out = np.zeros((rows.shape[0], d), dtype=np.float64)
    if scale is None:
        scale = 1.0 / np.sqrt(d)
    if nthreads is None:
        nthreads = os.cpu_count() or 1
    rc = _load().dar_oracle_attention(
        _DTYPES[dtype], B, int(Hq), Hkv, N, d, dd, int(w),
        _ptr(q_rows), _ptr(k), _ptr(v), _ptr(kd), _ptr(vd), _ptr(Uk), _ptr(Uv),
        float(scale), rows.shape[0], _ptr(rb), _ptr(rh), _ptr(ri), _ptr(out), int(nthreads))
    if rc != 0:
        raise ValueError("oracle rejected its arguments")
    return out


def prefill(q, k, v, Dk, Uk, Dv, Uv, w, dtype, scale=None, nthreads=None, rows=None):
    """Causal forward over positions 0..N-1 (the training-mode forward).

    ``q [B,Hq,N,d]``, ``k, v [B,Hkv,N,d]``.  With ``rows=None`` every position of
    every head is evaluated and f64 ``[B,Hq,N,d]`` is returned; otherwise only
    the ``(b, h, i)`` triples in ``rows`` are evaluated and f64 ``[R,d]`` is
    returned (sampled parity at large sizes)."""
    B, Hq, N, d = q.shape
    kd = down_project(k, Dk, dtype)
    vd = down_project(v, Dv, dtype)
    full = rows is None
    if full:
        bb, hh, ii = np.meshgrid(np.arange(B), np.arange(Hq), np.arange(N), indexing="ij")
        rows = np.stack([bb.ravel(), hh.ravel(), ii.ravel()], axis=1)
    rows = np.asarray(rows, dtype=np.int64).reshape(-1, 3)
    q_rows = np.ascontiguousarray(q[rows[:, 0], rows[:, 1], rows[:, 2]])
    out = attention_rows(q_rows, Hq, k, v, kd, vd, Uk, Uv, w, dtype, rows, scale, nthreads)
    return out.reshape(B, Hq, N, d) if full else out


def decode(q_last, k_hist, v_hist, lens, Dk, Uk, Dv, Uv, w, dtype, scale=None, nthreads=None,
           heads=None):
    """One inference step: the query of sequence b sits at position ``lens[b]-1``.

    ``q_last [B,Hq,d]``; ``k_hist, v_hist [B,Hkv,Nmax,d]`` hold the tokens of each
    sequence in order (only the first ``lens[b]`` are read).  Returns f64
    ``[B,Hq,d]``, zero where ``lens[b] == 0`` (no token to attend to).
    ``heads`` optionally restricts the evaluated ``(b, h)`` pairs."""
    B, Hq, d = q_last.shape
    lens = np.asarray(lens, dtype=np.int64)
    out = np.zeros((B, Hq, d), dtype=np.float64)
    if heads is None:
        heads = [(b, h) for b in range(B) for h in range(Hq)]
    by_seq = {}
    for b, h in heads:
        if lens[b] > 0:
            by_seq.setdefault(int(b), []).append(int(h))
    for b, hs in sorted(by_seq.items()):
        L = int(lens[b])
        kb = np.ascontiguousarray(k_hist[b:b + 1, :, :L])
        vb = np.ascontiguousarray(v_hist[b:b + 1, :, :L])
        kd = down_project(kb, Dk, dtype)
        vd = down_project(vb, Dv, dtype)
        rows = np.array([(0, h, L - 1) for h in hs], dtype=np.int32)
        q_rows = np.ascontiguousarray(q_last[b, hs])
        res = attention_rows(q_rows, Hq, kb, vb, kd, vd, Uk, Uv, w, dtype, rows, scale, nthreads)
        out[b, hs] = res
    return out


def attention_rows_direct(q_rows, qd_rows, Hq, k, v, kd, vd, Wo, w, dtype, rows, scale=None, scale_down=None,
                          nthreads=None):
    """Sec. 5, direct lower-dimensional global attention, for explicit rows.

    Local pairs (``i - j < w``, Eq. 3) score ``scale * q . k_j`` against the
    full-dimension keys; global pairs score ``scale_down * q^D . k^D_j`` in
    d_down, with ``qd_rows [R,dd]`` the d_down query of each row.  One softmax
    over both (Eq. 4); global values are ``v^D_j Wo`` with ``Wo [Hkv,dd,d]``.
    Defaults: ``scale = 1/sqrt(d)``, ``scale_down = 1/sqrt(dd)``.  Returns
    float64 ``[R,d]``."""
    q_rows, qd_rows, k, v, kd, vd = (_check(a, dtype) for a in (q_rows, qd_rows, k, v, kd, vd))
    Wo = np.ascontiguousarray(Wo, dtype=np.float32)
    B, Hkv, N, d = k.shape
    dd = kd.shape[3]
    rows = np.ascontiguousarray(rows, dtype=np.int32).reshape(-1, 3)
    assert q_rows.shape == (rows.shape[0], d) and qd_rows.shape == (rows.shape[0], dd)
    rb, rh, ri = (np.ascontiguousarray(rows[:, c]) for c in range(3))
    out = np.zeros((rows.shape[0], d), dtype=np.float64)
    scale = 1.0 / np.sqrt(d) if scale is None else scale
    scale_down = 1.0 / np.sqrt(dd) if scale_down is None else scale_down
    nthreads = (os.cpu_count() or 1) if nthreads is None else nthreads
    rc = _load().dar_oracle_attention_direct(
        _DTYPES[dtype], B, int(Hq), Hkv, N, d, dd, int(w),
        _ptr(q_rows), _ptr(qd_rows), _ptr(k), _ptr(v), _ptr(kd), _ptr(vd), _ptr(Wo),
        float(scale), float(scale_down), rows.shape[0], _ptr(rb), _ptr(rh), _ptr(ri), _ptr(out), int(nthreads))
    if rc != 0:
        raise ValueError("oracle rejected its arguments")
    return out


def prefill_direct(q, qd, k, v, Dk, Dv, Wo, w, dtype, scale=None, scale_down=None, nthreads=None, rows=None):
    """Causal forward of the direct variant over positions 0..N-1.

    ``q [B,Hq,N,d]``, ``qd [B,Hq,N,dd]`` (the d_down queries), ``k, v
    [B,Hkv,N,d]``; ``k^D, v^D`` come from Eq. 1 with ``Dk, Dv``.  Rows as in
    :func:`prefill`."""
    B, Hq, N, d = q.shape
    kd = down_project(k, Dk, dtype)
    vd = down_project(v, Dv, dtype)
    full = rows is None
    if full:
        bb, hh, ii = np.meshgrid(np.arange(B), np.arange(Hq), np.arange(N), indexing="ij")
        rows = np.stack([bb.ravel(), hh.ravel(), ii.ravel()], axis=1)
    rows = np.asarray(rows, dtype=np.int64).reshape(-1, 3)
    q_rows = np.ascontiguousarray(q[rows[:, 0], rows[:, 1], rows[:, 2]])
    qd_rows = np.ascontiguousarray(qd[rows[:, 0], rows[:, 1], rows[:, 2]])
    out = attention_rows_direct(q_rows, qd_rows, Hq, k, v, kd, vd, Wo, w, dtype, rows, scale, scale_down,
                                nthreads)
    return out.reshape(B, Hq, N, d) if full else out


def decode_direct(q_last, qd_last, k_hist, v_hist, lens, Dk, Dv, Wo, w, dtype, scale=None, scale_down=None,
                  nthreads=None, heads=None):
    """One inference step of the direct variant (query at ``lens[b]-1``).

    ``q_last [B,Hq,d]``, ``qd_last [B,Hq,dd]``; otherwise as :func:`decode`."""
    B, Hq, d = q_last.shape
    lens = np.asarray(lens, dtype=np.int64)
    out = np.zeros((B, Hq, d), dtype=np.float64)
    if heads is None:
        heads = [(b, h) for b in range(B) for h in range(Hq)]
    by_seq = {}
    for b, h in heads:
        if lens[b] > 0:
            by_seq.setdefault(int(b), []).append(int(h))
    for b, hs in sorted(by_seq.items()):
        L = int(lens[b])
        kb = np.ascontiguousarray(k_hist[b:b + 1, :, :L])
        vb = np.ascontiguousarray(v_hist[b:b + 1, :, :L])
        kd = down_project(kb, Dk, dtype)
        vd = down_project(vb, Dv, dtype)
        rows = np.array([(0, h, L - 1) for h in hs], dtype=np.int32)
        res = attention_rows_direct(np.ascontiguousarray(q_last[b, hs]), np.ascontiguousarray(qd_last[b, hs]), Hq,
                                    kb, vb, kd, vd, Wo, w, dtype, rows, scale, scale_down, nthreads)
        out[b, hs] = res
    return out


def backward(q, k, v, Dk, Uk, Dv, Uv, dout, w, dtype, scale=None, nthreads=None):
    """Sec. 2.3, training: gradients of the causal forward (:func:`prefill`)
    for the output gradient ``dout [B,Hq,N,d]`` (storage type).

    Returns a dict of float64 arrays: ``dq [B,Hq,N,d]``, ``dk, dv [B,Hkv,N,d]``,
    ``dDk, dDv [Hkv,d,dd]``, ``dUk, dUv [Hkv,dd,d]``.  The rounding of the
    stored ``k^D, v^D`` to the storage type is not differentiated."""
    q, k, v, dout = (_check(a, dtype) for a in (q, k, v, dout))
    Dk, Uk, Dv, Uv = (np.ascontiguousarray(a, dtype=np.float32) for a in (Dk, Uk, Dv, Uv))
    B, Hq, N, d = q.shape
    Hkv = k.shape[1]
    dd = Dk.shape[2]
    scale = 1.0 / np.sqrt(d) if scale is None else scale
    nthreads = (os.cpu_count() or 1) if nthreads is None else nthreads
    g = dict(dq=np.zeros((B, Hq, N, d)), dk=np.zeros((B, Hkv, N, d)), dv=np.zeros((B, Hkv, N, d)),
             dDk=np.zeros((Hkv, d, dd)), dUk=np.zeros((Hkv, dd, d)), dDv=np.zeros((Hkv, d, dd)),
             dUv=np.zeros((Hkv, dd, d)))
    rc = _load().dar_oracle_backward(
        _DTYPES[dtype], B, Hq, Hkv, N, d, dd, int(w), _ptr(q), _ptr(k), _ptr(v), _ptr(Dk), _ptr(Uk), _ptr(Dv),
        _ptr(Uv), _ptr(dout), float(scale), _ptr(g["dq"]), _ptr(g["dk"]), _ptr(g["dv"]), _ptr(g["dDk"]),
        _ptr(g["dUk"]), _ptr(g["dDv"]), _ptr(g["dUv"]), int(nthreads))
    if rc != 0:
        raise ValueError("oracle rejected its arguments")
    return g


def latent_rows(q_rows, Hq, k, v, c, Wup, WK, WV, w, dtype, rows, scale=None, nthreads=None):
    """Eq. 2-4 in the latent form for explicit rows ``(b, h, i)``.

    ``k, v [B,Hkv,N,d]`` the full keys/values (window branch of Eq. 3), ``c
    [B,N,dl]`` the stored bottleneck of every token (Eq. 1), ``Wup [dl,D]``,
    ``WK, WV [Hkv,D,d]``: distant keys/values are ``(c_j Wup) WK``, ``(c_j Wup)
    WV``, formed explicitly.  Returns float64 ``[R,d]``."""
    q_rows, k, v, c = (_check(a, dtype) for a in (q_rows, k, v, c))
    Wup, WK, WV = (np.ascontiguousarray(a, dtype=np.float32) for a in (Wup, WK, WV))
    B, Hkv, N, d = k.shape
    dl, D = Wup.shape
    assert c.shape == (B, N, dl) and WK.shape == (Hkv, D, d) and WV.shape == (Hkv, D, d)
    rows = np.ascontiguousarray(rows, dtype=np.int32).reshape(-1, 3)
    rb, rh, ri = (np.ascontiguousarray(rows[:, j]) for j in range(3))
    out = np.zeros((rows.shape[0], d), dtype=np.float64)
    scale = 1.0 / np.sqrt(d) if scale is None else scale
    nthreads = (os.cpu_count() or 1) if nthreads is None else nthreads
    rc = _load().dar_oracle_attention_latent(
        _DTYPES[dtype], B, int(Hq), Hkv, N, d, D, dl, int(w), _ptr(q_rows), _ptr(k), _ptr(v), _ptr(c), _ptr(Wup),
        _ptr(WK), _ptr(WV), float(scale), rows.shape[0], _ptr(rb), _ptr(rh), _ptr(ri), _ptr(out), int(nthreads))
    if rc != 0:
        raise ValueError("oracle rejected its arguments")
    return out


def latent_bottleneck(h, Wdown, dtype):
    """Eq. 1 on hidden states: ``h [B,n,D]`` times ``Wdown [D,dl]`` -> ``c [B,n,dl]``,
    each element one fp32 FMA chain over the D inputs, rounded to the storage
    type (the same chain as :func:`down_project`, with one shared bottleneck)."""
    return down_project(np.ascontiguousarray(h[:, None]), np.ascontiguousarray(Wdown[None]), dtype)[:, 0]


def latent_prefill(q, k, v, h, Wdown, Wup, WK, WV, w, dtype, scale=None, nthreads=None, rows=None):
    """Causal forward of the latent form over positions 0..N-1; ``h [B,N,D]``
    the hidden states the bottleneck is taken from (Eq. 1)."""
    B, Hq, N, d = q.shape
    c = latent_bottleneck(h, Wdown, dtype)
    full = rows is None
    if full:
        bb, hh, ii = np.meshgrid(np.arange(B), np.arange(Hq), np.arange(N), indexing="ij")
        rows = np.stack([bb.ravel(), hh.ravel(), ii.ravel()], axis=1)
    rows = np.asarray(rows, dtype=np.int64).reshape(-1, 3)
    q_rows = np.ascontiguousarray(q[rows[:, 0], rows[:, 1], rows[:, 2]])
    out = latent_rows(q_rows, Hq, k, v, c, Wup, WK, WV, w, dtype, rows, scale, nthreads)
    return out.reshape(B, Hq, N, d) if full else out


def latent_decode(q_last, k_hist, v_hist, h_hist, lens, Wdown, Wup, WK, WV, w, dtype, scale=None, nthreads=None,
                  heads=None):
    """One inference step of the latent form (query at ``lens[b]-1``):
    ``q_last [B,Hq,d]``, histories ``k_hist, v_hist [B,Hkv,Nmax,d]`` and
    ``h_hist [B,Nmax,D]`` (first ``lens[b]`` tokens read)."""
    B, Hq, d = q_last.shape
    lens = np.asarray(lens, dtype=np.int64)
    out = np.zeros((B, Hq, d), dtype=np.float64)
    if heads is None:
        heads = [(b, h) for b in range(B) for h in range(Hq)]
    by_seq = {}
    for b, h in heads:
        if lens[b] > 0:
            by_seq.setdefault(int(b), []).append(int(h))
    for b, hs in sorted(by_seq.items()):
        L = int(lens[b])
        c = latent_bottleneck(np.ascontiguousarray(h_hist[b:b + 1, :L]), Wdown, dtype)
        rows = np.array([(0, h, L - 1) for h in hs], dtype=np.int32)
        res = latent_rows(np.ascontiguousarray(q_last[b, hs]), Hq, np.ascontiguousarray(k_hist[b:b + 1, :, :L]),
                          np.ascontiguousarray(v_hist[b:b + 1, :, :L]), c, Wup, WK, WV, w, dtype, rows, scale,
                          nthreads)
        out[b, hs] = res
    return out
