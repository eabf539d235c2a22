"""C-ABI checks that need no GPU: the library builds for sm_103a, loads,
exports every function include/dar.h declares, and rejects bad arguments on
the host (error code, message, nothing launched)."""
import ctypes
import os
import shutil

import pytest

pytest.importorskip("torch")

from paper_2606_18587_gb300 import build as lib_build  # noqa: E402


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(lib_build.LIB) and shutil.which("nvcc") is None and \
            not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("no nvcc to build the library")
    lib_build.build()
    from paper_2606_18587_gb300 import dar
    return dar


def test_exports_every_declared_symbol(lib):
    names = lib.declared_symbols()
    assert {"dar_attn_prefill", "dar_attn_decode", "dar_cache_append", "dar_down_project",
            "dar_decode_workspace_bytes", "dar_prefill_workspace_bytes", "dar_last_error"} <= set(names)
    raw = ctypes.CDLL(lib.LIB_PATH)
    for n in names:
        assert hasattr(raw, n), f"{n} declared in dar.h but not exported"


def _cache(lib, **kw):
    c = dict(dtype=lib.DAR_BF16, B=2, Hkv=2, d=64, d_down=16, w=8, max_pages_per_seq=4, num_pages=8,
             win_k=256, win_v=512, pool_kd=768, pool_vd=1024, block_table=1280, seq_lens=1536, status=1792)
    c.update(kw)
    return lib.dar_cache(*[c[f] for f, _ in lib.dar_cache._fields_])


def test_workspace_sizes_are_host_only(lib):
    L = lib.load_library()
    c = _cache(lib)
    n = L.dar_decode_workspace_bytes(ctypes.byref(c), 4)
    assert n > 0 and n % 256 == 0
    assert L.dar_decode_workspace_bytes(ctypes.byref(c), 3) == 0      # Hq not a multiple of Hkv
    assert L.dar_decode_workspace_bytes(ctypes.byref(_cache(lib, d=32)), 4) == 0
    # k^D rows of 16 bf16 (2*3*100*16*2 B); v^D rows of 32 (16 values, then 16 ones for the row sums)
    assert L.dar_prefill_workspace_bytes(lib.DAR_BF16, 2, 3, 100, 16) == 19200 + 38400
    assert L.dar_prefill_workspace_bytes(lib.DAR_BF16, 1, 1, 4, 32) == 256 + 512   # rows of 32 and 64
    assert L.dar_prefill_workspace_bytes(lib.DAR_F32, 1, 1, 4, 32) == 2 * 512     # fp32: plain rows
    assert L.dar_prefill_workspace_bytes(lib.DAR_BF16, 1, 1, 3, 8) == 2 * 256  # 48 B rounded up to 256
    assert L.dar_prefill_workspace_bytes(lib.DAR_F32, 0, 3, 100, 16) == 0


def _a256(x):
    return (x + 255) // 256 * 256


@pytest.mark.parametrize("B,Hkv,Hq,dd", [(2, 2, 4, 16), (3, 8, 32, 16), (64, 8, 32, 64), (1, 1, 1, 8)])
def test_decode_workspace_layout(lib, B, Hkv, Hq, dd):
    """The decode workspace: q~ [B][Hq][dd] fp32, one counter per (sequence, KV
    head, head slice) group plus the pool's claim counter, and 2 slots x 2 types
    x GH records of 68 floats for each of the 160 x 8 warp ranges (no pool
    records while the pool is off) -- independent of the context capacity."""
    L = lib.load_library()
    G = Hq // Hkv
    GH = 4 if G % 4 == 0 else 2 if G % 2 == 0 else 1
    HS = G // GH
    want = _a256(B * Hq * dd * 4) + _a256((B * Hkv * HS + 1) * 4) + _a256(160 * 8 * 4 * GH * 68 * 4)
    for maxp in (1, 64, 4096):
        c = _cache(lib, B=B, Hkv=Hkv, d_down=dd, max_pages_per_seq=maxp, num_pages=B * maxp)
        assert L.dar_decode_workspace_bytes(ctypes.byref(c), Hq) == want
    # a small cache with four query heads per KV head fits the no-alloc entry point's scratch
    if B * Hq * dd * 4 < (1 << 20):
        assert want <= 8 << 20


@pytest.mark.parametrize("kw,code", [
    (dict(d=32), 2), (dict(d_down=12), 2), (dict(w=0), 1), (dict(Hkv=0), 1), (dict(dtype=7), 1),
    (dict(win_k=0), 1), (dict(win_k=258), 1), (dict(B=5000), 2), (dict(B=1025), 2),
])
def test_decode_rejects_bad_cache(lib, kw, code):
    L = lib.load_library()
    c = _cache(lib, **kw)
    r = L.dar_attn_decode(ctypes.byref(c), 4, 256, 256, 256, 0.0, 256, 256, 1 << 30, None)
    assert r == code
    assert L.dar_last_error().decode()


def test_prefill_rejects_bad_arguments(lib):
    L = lib.load_library()
    P = 4096
    args = lambda **kw: dict(dict(dtype=lib.DAR_BF16, B=1, Hq=4, Hkv=2, N=16, d=64, dd=16, w=4, q=P, k=P, v=P,  # noqa
                                   Dk=P, Uk=P, Dv=P, Uv=P, scale=0.0, out=P, ws=P, wsb=1 << 20, st=None, s=None),
                              **kw)

    def call(**kw):
        a = args(**kw)
        return L.dar_attn_prefill(a["dtype"], a["B"], a["Hq"], a["Hkv"], a["N"], a["d"], a["dd"], a["w"],
                                  a["q"], a["k"], a["v"], a["Dk"], a["Uk"], a["Dv"], a["Uv"], a["scale"],
                                  a["out"], a["ws"], a["wsb"], a["st"], a["s"])
    assert call(Hq=3) == 1
    assert call(w=-1) == 1
    assert call(d=128) == 2
    assert call(dd=24) == 2
    assert call(q=0) == 1
    assert call(k=P + 2) == 1
    assert call(wsb=16) == 3
    assert "workspace" in L.dar_last_error().decode()
    assert call(N=0) == 0          # empty problem: nothing to do
    assert L.dar_last_error().decode() == ""


def test_append_rejects_bad_arguments(lib):
    L = lib.load_library()
    c = _cache(lib)
    assert L.dar_cache_append(ctypes.byref(c), 256, 256, -1, None, 256, 256, None) == 1
    assert L.dar_cache_append(ctypes.byref(c), 0, 256, 4, None, 256, 256, None) == 1
    assert L.dar_cache_append(ctypes.byref(_cache(lib, w=0)), 256, 256, 4, None, 256, 256, None) == 1
    assert L.dar_cache_append(ctypes.byref(c), 256, 256, 0, None, 256, 256, None) == 0


def test_decode_step_checks_both_halves_before_launching(lib):
    """dar_decode_step refuses a bad append or a bad decode argument on the
    host (the same codes as the two calls alone), launching neither."""
    L = lib.load_library()
    c = _cache(lib)
    P = 4096

    def call(kn=P, n=1, Hq=4, q=P, ws=P, wsb=1 << 30, cache=c):
        return L.dar_decode_step(ctypes.byref(cache), kn, P, n, None, P, P, Hq, q, P, P, 0.0, P, ws, wsb, None)
    assert call(kn=0) == 1          # append: NULL k_new
    assert call(n=-1) == 1          # append: negative count
    assert call(Hq=3) == 1          # decode: Hq not a multiple of Hkv
    assert call(q=P + 8) == 1       # decode: misaligned query
    assert call(wsb=16) == 3        # decode: workspace too small
    assert "workspace" in L.dar_last_error().decode()
    assert call(cache=_cache(lib, d=32)) == 2


def test_bounded_wait_check_rejects_bad_arguments(lib):
    L = lib.load_library()
    assert L.dar_check_bounded_wait(None, 1000, None) == 1
    assert L.dar_check_bounded_wait(4096, 0, None) == 1
    assert L.dar_check_bounded_wait(4096, 2000001, None) == 1
    assert "limit_us" in L.dar_last_error().decode()


def _declared_param_counts(header):
    """Parameter count of every function declared in the header (C text)."""
    import re
    text = re.sub(r"/\*.*?\*/", "", open(header).read(), flags=re.S)
    counts = {}
    for m in re.finditer(r"\b(dar_\w+)\s*\(([^;{]*?)\)\s*;", text, re.S):
        params = m.group(2).strip()
        counts[m.group(1)] = 0 if params in ("", "void") else params.count(",") + 1
    return counts


def test_binding_argument_counts_match_the_header(lib):
    """Every ctypes signature in the Python binding has as many arguments as
    the C declaration it wraps."""
    L = lib.load_library()
    counts = _declared_param_counts(lib.HEADER)
    assert set(counts) == set(lib.declared_symbols())
    for name, n in counts.items():
        assert len(getattr(L, name).argtypes) == n, name


def test_direct_and_backward_reject_bad_arguments(lib):
    L = lib.load_library()
    P = 4096
    c = _cache(lib)
    # direct decode: NULL qd, misaligned qd, Hq not a multiple of Hkv
    assert L.dar_attn_decode_direct(ctypes.byref(c), 4, P, None, P, 0.0, 0.0, P, P, 1 << 30, None) == 1
    assert L.dar_attn_decode_direct(ctypes.byref(c), 4, P, P + 4, P, 0.0, 0.0, P, P, 1 << 30, None) == 1
    assert L.dar_attn_decode_direct(ctypes.byref(c), 3, P, P, P, 0.0, 0.0, P, P, 1 << 30, None) == 1
    # direct prefill: NULL qd, unsupported d_down
    pre = lambda qd=P, dd=16: L.dar_attn_prefill_direct(lib.DAR_BF16, 1, 4, 2, 16, 64, dd, 4, P, qd, P, P, P, P, P,  # noqa
                                                         0.0, 0.0, P, P, 1 << 20, None, None)
    assert pre(qd=None) == 1
    assert pre(dd=12) == 2

    # backward: workspace too small, NULL gradient, misaligned input
    def bwd(dq=P, k=P, wsb=1 << 40, Hq=4):
        return L.dar_attn_backward(lib.DAR_BF16, 1, Hq, 2, 16, 64, 16, 4, P, k, P, P, P, P, P, P, P, 0.0,
                                   dq, P, P, P, P, P, P, P, wsb, None)
    assert bwd(wsb=16) == 3
    assert bwd(dq=None) == 1
    assert bwd(k=P + 2) == 1
    assert bwd(Hq=3) == 1
    n = L.dar_attn_backward_workspace_bytes(lib.DAR_BF16, 1, 4, 2, 16, 16)
    assert n > 0 and n % 256 == 0
    assert L.dar_attn_backward_workspace_bytes(lib.DAR_BF16, 1, 3, 2, 16, 16) == 0


def _latent(lib, **kw):
    c = dict(B=2, Hkv=2, d=64, D=128, d_lat=64, w=8, max_pages_per_seq=4, num_pages=8, win_k=256, win_v=512,
             pool_c=768, block_table=1024, seq_lens=1280, status=1536)
    c.update(kw)
    return lib.dar_latent_cache(*[c[f] for f, _ in lib.dar_latent_cache._fields_])


def test_latent_entry_points_reject_bad_arguments(lib):
    """The latent form's entry points refuse bad shapes and pointers on the
    host, with the documented codes, and launch nothing."""
    L = lib.load_library()
    P = 4096
    c = _latent(lib)
    ws = L.dar_latent_decode_workspace_bytes(ctypes.byref(c), 4)
    assert ws > 0 and ws % 256 == 0
    assert L.dar_latent_decode_workspace_bytes(ctypes.byref(c), 3) == 0          # Hq not a multiple of Hkv
    assert L.dar_latent_decode_workspace_bytes(ctypes.byref(c), 34) == 0         # more than 32 query heads

    def dec(cache=c, Hq=4, q=P, wsb=1 << 30):
        return L.dar_latent_decode(ctypes.byref(cache), Hq, q, P, P, 0.0, P, P, wsb, None)
    assert dec(cache=_latent(lib, d_lat=96)) == 2     # d_lat not built
    assert dec(cache=_latent(lib, d=32)) == 2         # head dimension not built
    assert dec(cache=_latent(lib, B=1025)) == 2       # beyond the decode's batch limit
    assert dec(Hq=64) == 2                            # more than 32 query heads
    assert dec(Hq=3) == 1
    assert dec(q=0) == 1
    assert dec(q=P + 4) == 1                          # misaligned
    assert dec(wsb=16) == 3                           # workspace too small
    assert "workspace" in L.dar_last_error().decode()
    assert dec(cache=_latent(lib, B=0)) == 0          # nothing to do

    def app(cache=c, h=P, n=4, W=P):
        return L.dar_latent_append(ctypes.byref(cache), h, P, P, n, None, W, None)
    assert app(h=0) == 1
    assert app(n=-1) == 1
    assert app(W=P + 8) == 1
    assert app(cache=_latent(lib, D=8193)) == 2       # hidden width beyond the staging limit
    assert app(cache=_latent(lib, w=0)) == 1
    assert app(n=0) == 0

    assert L.dar_latent_absorb(2, 128, 32, 64, P, P, P, P, P, None) == 2   # d != 64
    assert L.dar_latent_absorb(0, 128, 64, 64, P, P, P, P, P, None) == 1   # no KV head
    assert L.dar_latent_absorb(2, 128, 64, 64, P, None, P, P, P, None) == 1


def test_chunk_and_down_project_reject_bad_arguments(lib):
    """dar_prefill_chunk (bf16, d_down >= 16) and dar_down_project refuse bad
    arguments on the host with the documented codes."""
    L = lib.load_library()
    P = 4096
    c = _cache(lib)
    n_ws = L.dar_prefill_chunk_workspace_bytes(ctypes.byref(c), 100)
    assert n_ws > 0 and n_ws % 256 == 0

    def chunk(cache=c, Hq=4, n=100, q=P, wsb=1 << 30):
        return L.dar_prefill_chunk(ctypes.byref(cache), Hq, n, q, P, P, P, P, P, P, 0.0, P, P, wsb, None)
    assert chunk(cache=_cache(lib, dtype=lib.DAR_F32)) == 2   # bf16 caches only
    assert chunk(cache=_cache(lib, d_down=8)) == 2            # d_down >= 16
    assert chunk(Hq=3) == 1
    assert chunk(n=-2) == 1
    assert chunk(q=P + 2) == 1
    assert chunk(wsb=16) == 3
    assert chunk(n=0) == 0

    def dp(B=1, n=10, d=64, dd=16, x=P, W=P, out=P):
        return L.dar_down_project(lib.DAR_BF16, B, 2, n, d, dd, x, W, out, None)
    assert dp(d=32) == 2
    assert dp(dd=12) == 2
    assert dp(n=-1) == 1
    assert dp(x=0) == 1
    assert dp(out=P + 2) == 1
    assert dp(n=0) == 0
