"""Seeded synthetic inputs for DAR attention.

Shared by the tests, the smoke check and the benchmark; it holds none of the
method's arithmetic.  Random numbers come from a counter-based generator:
splitmix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number
generators", OOPSLA 2014) keyed per (workload seed, tensor stream), mapped to
doubles in [0, 1) with the top 53 bits and to normals with the Box--Muller
transform.  Values are drawn in float64, rounded to float32 (nearest even) and,
for bfloat16 storage, rounded again to bfloat16 bit patterns (nearest even).
The generator's arithmetic is in ``inputs_gen.c`` (compiled with gcc on first use).

The paper trains on text corpora that are not available here; the workloads
below stand in for its attention shapes (head dim 64, d_down = d/4, windows of
about 128 to 512 tokens, contexts well past the window) with N(0, 1) queries,
keys and values, N(0, 1/d) down-projections and N(0, 1/d_down) up-projections.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_GEN_SRC = os.path.join(_HERE, "inputs_gen.c")
_GEN_LIB = os.path.join(_HERE, "libdar_inputs.so")
_gen = None

# tensor stream ids
S_Q, S_K, S_V, S_DK, S_DV, S_UK, S_UV, S_LENS, S_PAGES, S_QDEC, S_KNEW, S_VNEW, S_QD = range(1, 14)
S_H, S_WDOWN, S_WUP, S_WK, S_WV, S_HNEW = range(14, 20)
_KIND = {"f32": 0, "bf16": 1, "f64": 2, "uniform": 3}
_NP = {"f32": np.float32, "bf16": np.uint16, "f64": np.float64, "uniform": np.float64}


def build_generator(force: bool = False) -> str:
    """Compile the generator (gcc, no FMA contraction) next to this file."""
    if force or not os.path.exists(_GEN_LIB) or os.path.getmtime(_GEN_LIB) < os.path.getmtime(_GEN_SRC):
        tmp = _GEN_LIB + ".%d.tmp" % os.getpid()
        subprocess.run(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared", "-o", tmp,
                        _GEN_SRC, "-lm", "-lpthread"], check=True)
        os.replace(tmp, _GEN_LIB)
    return _GEN_LIB


def _lib():
    global _gen
    if _gen is None:
        lib = ctypes.CDLL(build_generator())
        lib.dargen_fill.argtypes = [ctypes.c_uint64] * 4 + [ctypes.c_size_t, ctypes.c_double, ctypes.c_int,
                                                            ctypes.c_void_p, ctypes.c_int]
        lib.dargen_fill.restype = None
        _gen = lib
    return _gen


def _fill(seed, stream, n, kind, std=1.0, sub=0, offset=0):
    out = np.empty(int(n), dtype=_NP[kind])
    if n:
        _lib().dargen_fill(seed, stream, sub, offset, int(n), float(std), _KIND[kind],
                           ctypes.c_void_p(out.ctypes.data), os.cpu_count() or 1)
    return out


def uniform(seed: int, stream: int, n: int, sub: int = 0, offset: int = 0) -> np.ndarray:
    """n doubles in [0, 1) from stream (seed, stream, sub), starting at element ``offset``."""
    return _fill(seed, stream, n, "uniform", sub=sub, offset=offset)


def normal(seed: int, stream: int, n: int, sub: int = 0) -> np.ndarray:
    """n standard normals in float64 (Box--Muller over consecutive uniform pairs)."""
    return _fill(seed, stream, n, "f64", sub=sub)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bfloat16 bit patterns, nearest even (inputs are finite)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))
    return (u >> np.uint64(16)).astype(np.uint16)


def bf16_bits_to_f32(h: np.ndarray) -> np.ndarray:
    return (np.asarray(h, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_array(seed, stream, shape, std=1.0, dtype="f32", sub=0) -> np.ndarray:
    """N(0, std^2) values drawn in float64 and rounded to the storage type."""
    n = int(np.prod(shape))
    return _fill(seed, stream, n, dtype, std=std, sub=sub).reshape(shape)


def projections(seed: int, Hkv: int, d: int, dd: int):
    """Dk, Dv ~ N(0, 1/d) of shape [Hkv,d,dd]; Uk, Uv ~ N(0, 1/dd) of shape [Hkv,dd,d]; float32."""
    Dk = normal_array(seed, S_DK, (Hkv, d, dd), std=1.0 / np.sqrt(d))
    Dv = normal_array(seed, S_DV, (Hkv, d, dd), std=1.0 / np.sqrt(d))
    Uk = normal_array(seed, S_UK, (Hkv, dd, d), std=1.0 / np.sqrt(dd))
    Uv = normal_array(seed, S_UV, (Hkv, dd, d), std=1.0 / np.sqrt(dd))
    return Dk, Uk, Dv, Uv


def latent_projections(seed: int, Hkv: int, D: int, dl: int, d: int):
    """The latent form's matrices, float32: Wdown [D,dl] ~ N(0, 1/D), Wup [dl,D]
    ~ N(0, 1/dl), WK, WV [Hkv,D,d] ~ N(0, 1/D) (unit-variance bottlenecks,
    lifted states and distant keys/values for unit-variance hidden states)."""
    Wdown = normal_array(seed, S_WDOWN, (D, dl), std=1.0 / np.sqrt(D))
    Wup = normal_array(seed, S_WUP, (dl, D), std=1.0 / np.sqrt(dl))
    WK = normal_array(seed, S_WK, (Hkv, D, d), std=1.0 / np.sqrt(D))
    WV = normal_array(seed, S_WV, (Hkv, D, d), std=1.0 / np.sqrt(D))
    return Wdown, Wup, WK, WV


# --------------------------------------------------------------------------- workloads


@dataclasses.dataclass(frozen=True)
class Prefill:
    name: str
    seed: int
    B: int
    Hq: int
    Hkv: int
    N: int
    d: int
    dd: int
    w: int
    dtype: str


@dataclasses.dataclass(frozen=True)
class Decode:
    name: str
    seed: int
    B: int
    Hq: int
    Hkv: int
    d: int
    dd: int
    w: int
    dtype: str
    L: Optional[int] = None          # uniform context length, or
    L_range: Optional[tuple] = None  # (lo, hi) inclusive, drawn per sequence
    shuffle_pages: bool = False      # physical page ids are a seeded permutation


PREFILL_TINY_F32 = Prefill("prefill-tiny-f32 B1 H4 N256 d64 dd16 w32", 1000, 1, 4, 4, 256, 64, 16, 32, "f32")
DECODE_160M = Decode("decode-160M bf16 B32 H12 L4096 d64 dd16 w128", 1001, 32, 12, 12, 64, 16, 128, "bf16", L=4096)
PREFILL_410M = Prefill("prefill-410M bf16 B8 H16 N8192 d64 dd16 w512", 1002, 8, 16, 16, 8192, 64, 16, 512, "bf16")
DECODE_1B_GQA = Decode("decode-1B-GQA paged bf16 B64 Hq32 Hkv8 L[1024,32768] d64 dd16 w256", 1003,
                       64, 32, 8, 64, 16, 256, "bf16", L_range=(1024, 32768), shuffle_pages=True)
SWEEP_W = (64, 256, 1024, 16384)
SWEEP_DD = (8, 16, 32, 64)


def sweep_point(k: int) -> Decode:
    """Point k (0..15) of the window x d_down decode sweep: B16 H16 L16384."""
    w = SWEEP_W[k // len(SWEEP_DD)]
    dd = SWEEP_DD[k % len(SWEEP_DD)]
    return Decode(f"decode-sweep bf16 B16 H16 L16384 w{w} dd{dd}", 1005 + k, 16, 16, 16, 64, dd, w,
                  "bf16", L=16384)


@dataclasses.dataclass(frozen=True)
class LatentDecode:
    """A decode workload of the latent form: hidden width D, bottleneck d_lat."""
    name: str
    seed: int
    B: int
    Hq: int
    Hkv: int
    d: int
    D: int
    dl: int
    w: int
    L: Optional[int] = None
    L_range: Optional[tuple] = None
    shuffle_pages: bool = False
    dtype: str = "bf16"


DECODE_160M_LATENT = LatentDecode("decode-160M-latent bf16 B32 H12 L4096 d64 D768 dlat192 w128", 1021,
                                  32, 12, 12, 64, 768, 192, 128, L=4096)
DECODE_1B_LATENT = LatentDecode("decode-1B-latent-GQA paged bf16 B64 Hq32 Hkv8 L[1024,8192] d64 D2048 dlat256 w256",
                                1023, 64, 32, 8, 64, 2048, 256, 256, L_range=(1024, 8192), shuffle_pages=True)


def latent_history(cfg: LatentDecode, b: int, L: Optional[int] = None):
    """Hidden states [L, D] and keys/values [Hkv, L, d] of every token of
    sequence b, N(0, 1) in the storage type (one stream per sequence)."""
    if L is None:
        L = int(decode_lengths(cfg)[b])
    h = normal_array(cfg.seed, S_H, (L, cfg.D), dtype=cfg.dtype, sub=b + 1)
    k = normal_array(cfg.seed, S_K, (cfg.Hkv, L, cfg.d), dtype=cfg.dtype, sub=b + 1)
    v = normal_array(cfg.seed, S_V, (cfg.Hkv, L, cfg.d), dtype=cfg.dtype, sub=b + 1)
    return h, k, v


def prefill_inputs(cfg: Prefill):
    """q [B,Hq,N,d], k, v [B,Hkv,N,d] (storage type) and the four projections."""
    s = cfg.seed
    q = normal_array(s, S_Q, (cfg.B, cfg.Hq, cfg.N, cfg.d), dtype=cfg.dtype)
    k = normal_array(s, S_K, (cfg.B, cfg.Hkv, cfg.N, cfg.d), dtype=cfg.dtype)
    v = normal_array(s, S_V, (cfg.B, cfg.Hkv, cfg.N, cfg.d), dtype=cfg.dtype)
    Dk, Uk, Dv, Uv = projections(s, cfg.Hkv, cfg.d, cfg.dd)
    return dict(q=q, k=k, v=v, Dk=Dk, Uk=Uk, Dv=Dv, Uv=Uv)


def direct_queries(cfg, step: int = 0) -> np.ndarray:
    """The d_down queries of the direct global path (Sec. 5), N(0, 1) in the
    storage type: [B, Hq, N, dd] for a prefill config, [B, Hq, dd] for a decode
    config (at one decode step)."""
    if isinstance(cfg, Prefill):
        return normal_array(cfg.seed, S_QD, (cfg.B, cfg.Hq, cfg.N, cfg.dd), dtype=cfg.dtype)
    return normal_array(cfg.seed, S_QD, (cfg.B, cfg.Hq, cfg.dd), dtype=cfg.dtype, sub=step)


def decode_lengths(cfg: Decode) -> np.ndarray:
    """Context length of each sequence (int64 [B])."""
    if cfg.L is not None:
        return np.full(cfg.B, cfg.L, dtype=np.int64)
    lo, hi = cfg.L_range
    u = uniform(cfg.seed, S_LENS, cfg.B)
    return lo + np.floor(u * (hi - lo + 1)).astype(np.int64)


def decode_history(cfg: Decode, b: int, L: Optional[int] = None):
    """Keys and values of every token of sequence b, in order: two [Hkv, L, d] arrays.

    Each sequence has its own stream, so one sequence can be generated alone."""
    if L is None:
        L = int(decode_lengths(cfg)[b])
    k = normal_array(cfg.seed, S_K, (cfg.Hkv, L, cfg.d), dtype=cfg.dtype, sub=b + 1)
    v = normal_array(cfg.seed, S_V, (cfg.Hkv, L, cfg.d), dtype=cfg.dtype, sub=b + 1)
    return k, v


def decode_query(cfg: Decode, step: int = 0) -> np.ndarray:
    """The query of each sequence at one decode step: [B, Hq, d] (storage type)."""
    return normal_array(cfg.seed, S_QDEC, (cfg.B, cfg.Hq, cfg.d), dtype=cfg.dtype, sub=step)


def decode_new_tokens(cfg: Decode, step: int = 0):
    """Key/value of the token each sequence appends at one decode step: two [B, Hkv, 1, d]."""
    k = normal_array(cfg.seed, S_KNEW, (cfg.B, cfg.Hkv, 1, cfg.d), dtype=cfg.dtype, sub=step)
    v = normal_array(cfg.seed, S_VNEW, (cfg.B, cfg.Hkv, 1, cfg.d), dtype=cfg.dtype, sub=step)
    return k, v


def page_assignment(cfg: Decode, capacity_tokens: np.ndarray, page_size: int = 64):
    """Block table for a paged cache: sequence b gets ceil(cap_b / page_size) pages.

    Returns (block_table int32 [B, max_pages_per_seq] with -1 for unassigned
    slots, num_pages).  With ``cfg.shuffle_pages`` the physical ids are a seeded
    permutation; otherwise they are handed out in order."""
    cap = np.asarray(capacity_tokens, dtype=np.int64)
    npages = (np.maximum(cap, 0) + page_size - 1) // page_size
    total = int(npages.sum())
    maxp = max(1, int(npages.max()) if len(npages) else 1)
    if cfg.shuffle_pages:
        ids = np.argsort(uniform(cfg.seed, S_PAGES, total), kind="stable").astype(np.int32)
    else:
        ids = np.arange(total, dtype=np.int32)
    table = np.full((len(cap), maxp), -1, dtype=np.int32)
    off = 0
    for b, n in enumerate(npages):
        table[b, :n] = ids[off:off + n]
        off += n
    return table, max(total, 1)
