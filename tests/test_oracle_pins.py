"""Pins for the CPU oracle: each test checks it against something other than itself.

Sources of truth: closed forms of Eq. 1-4, a textbook attention written here
independently, torch's scaled_dot_product_attention (float64, CPU), exact
rational arithmetic, a 50-digit mpmath evaluation, and the numbers the paper
prints in Table 1 / Table 3 (tests/golden/window_ablation_w0.txt).
"""
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2606_18587_gb300 import inputs as I

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------------------- helpers


def rand_case(seed, B, Hq, Hkv, N, d, dd, dtype="f32"):
    q = I.normal_array(seed, I.S_Q, (B, Hq, N, d), dtype=dtype)
    k = I.normal_array(seed, I.S_K, (B, Hkv, N, d), dtype=dtype)
    v = I.normal_array(seed, I.S_V, (B, Hkv, N, d), dtype=dtype)
    Dk, Uk, Dv, Uv = I.projections(seed, Hkv, d, dd)
    return q, k, v, Dk, Uk, Dv, Uv


def textbook_causal(q, keys, vals, scale):
    """softmax(scale * q K^T, causal) V for one head; q [N,d], keys/vals [N,d] float64."""
    N = q.shape[0]
    s = scale * (q @ keys.T)
    s[np.triu_indices(N, 1)] = -np.inf
    s -= s.max(axis=1, keepdims=True)
    p = np.exp(s)
    p /= p.sum(axis=1, keepdims=True)
    return p @ vals


def f64(a, dtype):
    return oracle.to_f64(a, dtype)


def round_f32_exact(x: Fraction) -> Fraction:
    """Nearest float32 to a rational, ties to even (exact search over neighbours)."""
    c = np.float32(float(x))
    cands = {c, np.nextafter(c, np.float32(np.inf)), np.nextafter(c, np.float32(-np.inf))}
    best = None
    for v in cands:
        err = abs(Fraction(float(v)) - x)
        even = (int(np.array(v, dtype=np.float32).view(np.uint32)) & 1) == 0
        key = (err, not even)
        if best is None or key < best[0]:
            best = (key, v)
    return Fraction(float(best[1]))


def round_bf16_bits_exact(x: float) -> int:
    """bfloat16 bits nearest to a float32 value, ties to even, via exact distances."""
    u = int(np.array(x, dtype=np.float32).view(np.uint32))
    lo = u >> 16
    best = None
    for h in (lo, lo + 1):
        val = float(np.array(h << 16, dtype=np.uint32).view(np.float32))
        err = abs(Fraction(val) - Fraction(float(x)))
        key = (err, h & 1)
        if best is None or key < best[0]:
            best = (key, h)
    return best[1]


# ----------------------------------------------------------------------------- Eq. 1


def test_bf16_rounding_matches_exact_nearest_even():
    rng = np.random.default_rng(5)
    vals = rng.standard_normal(4000).astype(np.float32)
    # exact ties: bit 15 set, low 15 bits clear, both parities of bit 16
    ties = np.array([0x3F808000, 0x3F818000, 0xBF808000, 0x40490000 | 0x8000], dtype=np.uint32).view(np.float32)
    vals = np.concatenate([vals, ties])
    got = oracle.f32_to_bf16(vals)
    want = np.array([round_bf16_bits_exact(float(v)) for v in vals], dtype=np.uint16)
    np.testing.assert_array_equal(got, want)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_down_projection_is_the_exact_fp32_fma_chain(dtype):
    """Eq. 1 element = round_T(fmaf chain over t = 0..d-1 from +0), checked in exact rationals."""
    B, Hkv, n, d, dd = 1, 2, 3, 8, 4
    x = I.normal_array(11, I.S_K, (B, Hkv, n, d), dtype=dtype)
    Dw = I.normal_array(11, I.S_DK, (Hkv, d, dd), std=1 / np.sqrt(d))
    got = oracle.down_project(x, Dw, dtype)
    xf = f64(x, dtype)
    for b in range(B):
        for g in range(Hkv):
            for j in range(n):
                for c in range(dd):
                    acc = Fraction(0)
                    for t in range(d):
                        acc = round_f32_exact(Fraction(float(xf[b, g, j, t])) * Fraction(float(Dw[g, t, c])) + acc)
                    if dtype == "f32":
                        assert Fraction(float(got[b, g, j, c])) == acc
                    else:
                        assert int(got[b, g, j, c]) == round_bf16_bits_exact(float(acc))


def test_down_projection_close_to_matmul():
    """Same operand orientation as x @ W_down (a transposed Dw would fail)."""
    x = I.normal_array(3, I.S_K, (2, 3, 50, 64))
    Dw = I.normal_array(3, I.S_DK, (3, 64, 16), std=1 / 8)
    got = oracle.down_project(x, Dw, "f32").astype(np.float64)
    want = np.einsum("bgnt,gtc->bgnc", x.astype(np.float64), Dw.astype(np.float64))
    np.testing.assert_allclose(got, want, rtol=0, atol=5e-6)


# ----------------------------------------------------------------------------- Eq. 2-4


@pytest.mark.parametrize("extra", [0, 7])
def test_P1_window_covering_everything_is_causal_attention(extra):
    torch = pytest.importorskip("torch")
    B, H, N, d, dd = 2, 3, 40, 16, 4
    q, k, v, Dk, Uk, Dv, Uv = rand_case(21, B, H, H, N, d, dd)
    got = oracle.prefill(q, k, v, Dk, Uk, Dv, Uv, w=N + extra, dtype="f32")
    scale = 1 / np.sqrt(d)
    for b in range(B):
        for h in range(H):
            want = textbook_causal(f64(q[b, h], "f32"), f64(k[b, h], "f32"), f64(v[b, h], "f32"), scale)
            np.testing.assert_allclose(got[b, h], want, rtol=0, atol=1e-12)
    sdpa = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q.astype(np.float64)), torch.from_numpy(k.astype(np.float64)),
        torch.from_numpy(v.astype(np.float64)), is_causal=True).numpy()
    np.testing.assert_allclose(got, sdpa, rtol=0, atol=1e-12)


def test_P2_identity_bottleneck_is_full_attention():
    B, H, N, d = 1, 2, 33, 16
    q, k, v, _, _, _, _ = rand_case(22, B, H, H, N, d, d, dtype="bf16")
    eye = np.broadcast_to(np.eye(d, dtype=np.float32), (H, d, d)).copy()
    # the stored bottleneck is bit-identical to the input
    np.testing.assert_array_equal(oracle.down_project(k, eye, "bf16"), k)
    got = oracle.prefill(q, k, v, eye, eye, eye, eye, w=5, dtype="bf16")
    for h in range(H):
        want = textbook_causal(f64(q[0, h], "bf16"), f64(k[0, h], "bf16"), f64(v[0, h], "bf16"), 1 / np.sqrt(d))
        np.testing.assert_allclose(got[0, h], want, rtol=0, atol=1e-12)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_P3_zero_window_is_uniform_reduction(dtype):
    """w = 0: every key/value, the current token's included, comes from h^D W_up."""
    B, Hq, Hkv, N, d, dd = 1, 4, 2, 30, 16, 4
    q, k, v, Dk, Uk, Dv, Uv = rand_case(23, B, Hq, Hkv, N, d, dd, dtype)
    got = oracle.prefill(q, k, v, Dk, Uk, Dv, Uv, w=0, dtype=dtype)
    kd = f64(oracle.down_project(k, Dk, dtype), dtype)
    vd = f64(oracle.down_project(v, Dv, dtype), dtype)
    for h in range(Hq):
        g = h // (Hq // Hkv)
        klift = kd[0, g] @ Uk[g].astype(np.float64)
        vlift = vd[0, g] @ Uv[g].astype(np.float64)
        want = textbook_causal(f64(q[0, h], dtype), klift, vlift, 1 / np.sqrt(d))
        np.testing.assert_allclose(got[0, h], want, rtol=0, atol=1e-12)


def test_P4_zero_lift_gives_closed_form():
    """Uk = Uv = 0: every global token has score 0 and value 0, so
    o_i = sum_loc e^{s_j} v_j / (sum_loc e^{s_j} + max(0, i + 1 - w))."""
    B, H, N, d, dd, w = 1, 2, 50, 16, 4, 9
    q, k, v, Dk, Uk, Dv, Uv = rand_case(24, B, H, H, N, d, dd)
    zero = np.zeros_like(Uk)
    got = oracle.prefill(q, k, v, Dk, zero, Dv, zero, w=w, dtype="f32")
    for h in range(H):
        qq, kk, vv = (f64(a[0, h], "f32") for a in (q, k, v))
        for i in range(N):
            js = np.arange(max(0, i - w + 1), i + 1)
            e = np.exp(qq[i] @ kk[js].T / np.sqrt(d))
            want = (e @ vv[js]) / (e.sum() + max(0, i + 1 - w))
            np.testing.assert_allclose(got[0, h, i], want, rtol=0, atol=1e-12)


def test_P5_causality_bit_identical():
    B, H, N, d, dd, w = 1, 2, 24, 16, 4, 5
    q, k, v, Dk, Uk, Dv, Uv = rand_case(25, B, H, H, N, d, dd)
    base = oracle.prefill(q, k, v, Dk, Uk, Dv, Uv, w=w, dtype="f32")
    i = 13
    k2, v2 = k.copy(), v.copy()
    k2[:, :, i + 1:] += 3.0
    v2[:, :, i + 1:] -= 2.0
    pert = oracle.prefill(q, k2, v2, Dk, Uk, Dv, Uv, w=w, dtype="f32")
    np.testing.assert_array_equal(pert[:, :, :i + 1], base[:, :, :i + 1])
    assert not np.array_equal(pert[:, :, i + 1:], base[:, :, i + 1:])


def test_P6_window_edge():
    """For query i: token i-w+1 is read only through its full vectors, token i-w
    only through its bottleneck vectors (Eq. 3 with local iff i - j < w)."""
    B, H, N, d, dd, w = 1, 1, 20, 16, 4, 6
    q, k, v, Dk, Uk, Dv, Uv = rand_case(26, B, H, H, N, d, dd)
    kd = oracle.down_project(k, Dk, "f32")
    vd = oracle.down_project(v, Dv, "f32")
    i = 15
    rows = np.array([[0, 0, i]])
    qr = np.ascontiguousarray(q[0, 0, [i]])

    def run(k_, v_, kd_, vd_):
        return oracle.attention_rows(qr, H, k_, v_, kd_, vd_, Uk, Uv, w, "f32", rows)

    base = run(k, v, kd, vd)
    inside, outside = i - w + 1, i - w

    def bumped(a, j):
        a = a.copy()
        a[0, 0, j] += 1.5
        return a

    # changes that must not matter
    np.testing.assert_array_equal(run(k, v, bumped(kd, inside), bumped(vd, inside)), base)
    np.testing.assert_array_equal(run(bumped(k, outside), bumped(v, outside), kd, vd), base)
    # changes that must matter
    assert not np.array_equal(run(k, v, bumped(kd, outside), vd), base)
    assert not np.array_equal(run(k, v, kd, bumped(vd, outside)), base)
    assert not np.array_equal(run(bumped(k, inside), v, kd, vd), base)
    assert not np.array_equal(run(k, bumped(v, inside), kd, vd), base)


def test_P7_absorption_identity():
    """The GPU scores distant keys as (q Uk^T) . k^D and lifts sum_j p_j v^D_j once;
    both equal the explicit Eq. 2 lift by linearity."""
    rng = np.random.default_rng(7)
    d, dd, n = 64, 16, 300
    q = rng.standard_normal(d)
    kd = rng.standard_normal((n, dd))
    vd = rng.standard_normal((n, dd))
    Uk = rng.standard_normal((dd, d)) / 4
    Uv = rng.standard_normal((dd, d)) / 4
    p = rng.random(n)
    np.testing.assert_allclose((q @ Uk.T) @ kd.T, q @ (kd @ Uk).T, rtol=0, atol=1e-12)
    np.testing.assert_allclose((p @ vd) @ Uv, p @ (vd @ Uv), rtol=0, atol=1e-12)


def test_P8_mpmath_brute_force():
    mp = pytest.importorskip("mpmath")
    mp.mp.dps = 50
    B, Hq, Hkv, N, d, dd, w = 1, 2, 1, 7, 4, 2, 3
    q, k, v, Dk, Uk, Dv, Uv = rand_case(28, B, Hq, Hkv, N, d, dd)
    got = oracle.prefill(q, k, v, Dk, Uk, Dv, Uv, w=w, dtype="f32")
    kd = oracle.down_project(k, Dk, "f32")
    vd = oracle.down_project(v, Dv, "f32")
    M = lambda x: mp.mpf(float(x))  # noqa: E731
    for h in range(Hq):
        for i in range(N):
            s, vals = [], []
            for j in range(i + 1):
                if i - j < w:
                    key = [M(k[0, 0, j, t]) for t in range(d)]
                    val = [M(v[0, 0, j, t]) for t in range(d)]
                else:
                    key = [sum(M(kd[0, 0, j, c]) * M(Uk[0, c, t]) for c in range(dd)) for t in range(d)]
                    val = [sum(M(vd[0, 0, j, c]) * M(Uv[0, c, t]) for c in range(dd)) for t in range(d)]
                s.append(sum(M(q[0, h, i, t]) * key[t] for t in range(d)) / mp.sqrt(d))
                vals.append(val)
            z = sum(mp.exp(x) for x in s)
            for t in range(d):
                o = sum(mp.exp(s[j]) * vals[j][t] for j in range(i + 1)) / z
                assert abs(float(o) - got[0, h, i, t]) < 1e-12


def test_gqa_head_mapping_matches_repeated_kv():
    """Query head h reads KV head h // (Hq/Hkv): same as MHA with each KV head repeated."""
    B, Hq, Hkv, N, d, dd, w = 1, 6, 2, 20, 16, 4, 4
    q, k, v, Dk, Uk, Dv, Uv = rand_case(29, B, Hq, Hkv, N, d, dd)
    got = oracle.prefill(q, k, v, Dk, Uk, Dv, Uv, w=w, dtype="f32")
    rep = lambda a: np.ascontiguousarray(np.repeat(a, Hq // Hkv, axis=0))  # noqa: E731
    krep = np.ascontiguousarray(np.repeat(k, Hq // Hkv, axis=1))
    vrep = np.ascontiguousarray(np.repeat(v, Hq // Hkv, axis=1))
    want = oracle.prefill(q, krep, vrep, rep(Dk), rep(Uk), rep(Dv), rep(Uv), w=w, dtype="f32")
    np.testing.assert_array_equal(got, want)
    # and not the other (h % Hkv) mapping
    alt = [h % Hkv for h in range(Hq)]
    want_alt = oracle.prefill(q, np.ascontiguousarray(k[:, alt]), np.ascontiguousarray(v[:, alt]),
                              Dk[alt].copy(), Uk[alt].copy(), Dv[alt].copy(), Uv[alt].copy(), w=w, dtype="f32")
    assert not np.allclose(got, want_alt)


def test_decode_is_last_prefill_row():
    B, Hq, Hkv, d, dd, w = 3, 4, 2, 16, 4, 5
    lens = np.array([1, 9, 14])
    Nmax = 14
    q, k, v, Dk, Uk, Dv, Uv = rand_case(30, B, Hq, Hkv, Nmax, d, dd, dtype="bf16")
    qlast = np.ascontiguousarray(np.stack([q[b, :, lens[b] - 1] for b in range(B)]))
    got = oracle.decode(qlast, k, v, lens, Dk, Uk, Dv, Uv, w, "bf16")
    full = oracle.prefill(q, k, v, Dk, Uk, Dv, Uv, w=w, dtype="bf16")
    for b in range(B):
        np.testing.assert_allclose(got[b], full[b, :, lens[b] - 1], rtol=0, atol=1e-13)
    # no token at all: zero output by convention
    z = oracle.decode(qlast, k, v, np.array([0, 9, 14]), Dk, Uk, Dv, Uv, w, "bf16")
    assert np.all(z[0] == 0)


def test_golden_window_ablation_pins_boundary_reading():
    """Table 3's w = 0 row equals Table 1's uniform-reduction row (no local token at
    w = 0); w = 1 differs (the current token is local)."""
    rows = {}
    for line in open(os.path.join(GOLDEN, "window_ablation_w0.txt")):
        if line.strip() and not line.startswith("#"):
            key, *vals = line.split()
            rows[key] = [float(x) for x in vals]
    assert rows["w0"] == rows["uniform_dd128"]
    assert rows["w1"] != rows["w0"]
    # The oracle implements exactly that reading:
    B, H, N, d, dd = 1, 1, 12, 8, 2
    q, k, v, Dk, Uk, Dv, Uv = rand_case(31, B, H, H, N, d, dd)
    kd = f64(oracle.down_project(k, Dk, "f32"), "f32")[0, 0]
    vd = f64(oracle.down_project(v, Dv, "f32"), "f32")[0, 0]
    klift, vlift = kd @ Uk[0].astype(np.float64), vd @ Uv[0].astype(np.float64)
    qq, kk, vv = (f64(a[0, 0], "f32") for a in (q, k, v))
    got1 = oracle.prefill(q, k, v, Dk, Uk, Dv, Uv, w=1, dtype="f32")[0, 0]
    for i in range(N):
        keys = klift[: i + 1].copy()
        vals = vlift[: i + 1].copy()
        keys[i], vals[i] = kk[i], vv[i]      # w = 1: only the current token is local
        s = qq[i] @ keys.T / np.sqrt(d)
        p = np.exp(s - s.max())
        np.testing.assert_allclose(got1[i], p @ vals / p.sum(), rtol=0, atol=1e-12)


def test_rejects_bad_arguments():
    q, k, v, Dk, Uk, Dv, Uv = rand_case(32, 1, 2, 2, 8, 8, 2)
    kd = oracle.down_project(k, Dk, "f32")
    vd = oracle.down_project(v, Dv, "f32")
    with pytest.raises(ValueError):
        oracle.attention_rows(np.ascontiguousarray(q[0, 0, :1]), 2, k, v, kd, vd, Uk, Uv, 2, "f32",
                              np.array([[0, 0, 8]]))  # position out of range
    with pytest.raises(ValueError):
        oracle.attention_rows(np.ascontiguousarray(q[0, 0, :1]), 2, k, v, kd, vd, Uk, Uv, -1, "f32",
                              np.array([[0, 0, 3]]))  # negative window
