"""Pins for the latent-form oracle (oracle.latent_rows / latent_prefill /
latent_decode: Eq. 1-4 on hidden states with one bottleneck per token shared
by every head, keys and values).  Each test checks it against something other
than itself: the per-head oracle (pinned in test_oracle_pins.py) where the two
forms coincide, torch's scaled_dot_product_attention in float64 where the
method reduces to attention over fixed keys, and invariants of Eq. 3."""
import numpy as np
import pytest

import oracle
from paper_2606_18587_gb300 import inputs as I

torch = pytest.importorskip("torch")


def case(seed, B=2, Hq=4, Hkv=2, N=40, d=16, D=24, dl=8, dtype="f32"):
    q = I.normal_array(seed, I.S_Q, (B, Hq, N, d), dtype=dtype)
    k = I.normal_array(seed, I.S_K, (B, Hkv, N, d), dtype=dtype)
    v = I.normal_array(seed, I.S_V, (B, Hkv, N, d), dtype=dtype)
    h = I.normal_array(seed, I.S_H, (B, N, D), dtype=dtype)
    Wdown, Wup, WK, WV = I.latent_projections(seed, Hkv, D, dl, d)
    return q, k, v, h, Wdown, Wup, WK, WV


def sdpa(q, k, v, scale):
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a))[None, None]
    return torch.nn.functional.scaled_dot_product_attention(t(q), t(k), t(v), is_causal=True,
                                                            scale=scale)[0, 0].numpy()


@pytest.mark.parametrize("w", [0, 1, 9, 40])
def test_identity_key_value_maps_give_the_per_head_form(w):
    """D = d and W_K = W_V = I: distant keys and values are c_j W_up, which is
    the per-head method with k^D = v^D = c and Uk = Uv = W_up."""
    q, k, v, h, Wdown, Wup, _, _ = case(51, D=16)
    Hkv, d = k.shape[1], k.shape[3]
    eye = np.broadcast_to(np.eye(d, dtype=np.float32), (Hkv, d, d)).copy()
    got = oracle.latent_prefill(q, k, v, h, Wdown, Wup, eye, eye, w, "f32")
    c = oracle.latent_bottleneck(h, Wdown, "f32")
    cg = np.ascontiguousarray(np.broadcast_to(c[:, None], (c.shape[0], Hkv) + c.shape[1:]))
    U = np.ascontiguousarray(np.broadcast_to(Wup, (Hkv,) + Wup.shape))
    B, Hq, N, _ = q.shape
    bb, hh, ii = np.meshgrid(np.arange(B), np.arange(Hq), np.arange(N), indexing="ij")
    rows = np.stack([bb.ravel(), hh.ravel(), ii.ravel()], axis=1)
    want = oracle.attention_rows(np.ascontiguousarray(q[rows[:, 0], rows[:, 1], rows[:, 2]]), Hq, k, v, cg, cg,
                                 U, U, w, "f32", rows).reshape(B, Hq, N, d)
    assert np.abs(got - want).max() < 1e-12


def test_window_covering_everything_is_causal_attention():
    q, k, v, h, Wdown, Wup, WK, WV = case(52)
    N, d = q.shape[2], q.shape[3]
    got = oracle.latent_prefill(q, k, v, h, Wdown, Wup, WK, WV, N, "f32")
    G = q.shape[1] // k.shape[1]
    for b in range(q.shape[0]):
        for hq in range(q.shape[1]):
            want = sdpa(q[b, hq].astype(np.float64), k[b, hq // G].astype(np.float64),
                        v[b, hq // G].astype(np.float64), 1 / np.sqrt(d))
            assert np.abs(got[b, hq] - want).max() < 1e-12


def test_zero_window_is_attention_on_lifted_keys():
    """w = 0: every pair takes (c_j W_up) W_K, (c_j W_up) W_V (numpy matmuls
    on the stored bottleneck), then plain causal attention."""
    q, k, v, h, Wdown, Wup, WK, WV = case(53, dtype="bf16")
    d = q.shape[3]
    got = oracle.latent_prefill(q, k, v, h, Wdown, Wup, WK, WV, 0, "bf16")
    c = oracle.to_f64(oracle.latent_bottleneck(h, Wdown, "bf16"), "bf16")
    G = q.shape[1] // k.shape[1]
    for b in range(q.shape[0]):
        hl = c[b] @ Wup.astype(np.float64)
        for hq in range(q.shape[1]):
            g = hq // G
            want = sdpa(oracle.to_f64(q[b, hq], "bf16"), hl @ WK[g].astype(np.float64),
                        hl @ WV[g].astype(np.float64), 1 / np.sqrt(d))
            assert np.abs(got[b, hq] - want).max() < 1e-12


def test_window_edge():
    """Row i reads the bottleneck only of tokens j <= i - w and the full keys
    only of tokens j > i - w (Eq. 3): perturbing the other representation of a
    token leaves the row bit-identical."""
    q, k, v, h, Wdown, Wup, WK, WV = case(54, B=1, Hq=2, Hkv=1, N=30)
    w, i = 6, 20
    base = oracle.latent_prefill(q, k, v, h, Wdown, Wup, WK, WV, w, "f32")[0, :, i]
    h2 = h.copy()
    h2[0, i - w + 1:] += 1.0      # bottlenecks of the window tokens and later ones
    k2, v2 = k.copy(), v.copy()
    k2[0, :, :i - w + 1] += 1.0  # full keys/values of the distant tokens
    v2[0, :, :i - w + 1] += 1.0
    assert np.array_equal(base, oracle.latent_prefill(q, k, v, h2, Wdown, Wup, WK, WV, w, "f32")[0, :, i])
    assert np.array_equal(base, oracle.latent_prefill(q, k2, v2, h, Wdown, Wup, WK, WV, w, "f32")[0, :, i])
    h3 = h.copy()
    h3[0, i - w] += 1.0            # the newest distant token does matter
    assert not np.array_equal(base, oracle.latent_prefill(q, k, v, h3, Wdown, Wup, WK, WV, w, "f32")[0, :, i])


def test_decode_is_the_last_prefill_row():
    q, k, v, h, Wdown, Wup, WK, WV = case(55, B=2, N=33, dtype="bf16")
    lens = [33, 21]
    q_last = np.stack([q[b, :, lens[b] - 1] for b in range(2)])
    got = oracle.latent_decode(q_last, k, v, h, lens, Wdown, Wup, WK, WV, 7, "bf16")
    for b in range(2):
        L = lens[b]
        full = oracle.latent_prefill(np.ascontiguousarray(q[b:b + 1, :, :L]), np.ascontiguousarray(k[b:b + 1, :, :L]),
                                     np.ascontiguousarray(v[b:b + 1, :, :L]), np.ascontiguousarray(h[b:b + 1, :L]),
                                     Wdown, Wup, WK, WV, 7, "bf16")
        assert np.array_equal(got[b], full[0, :, L - 1])


def test_bottleneck_is_the_hidden_state_times_w_down():
    """Eq. 1 on hidden states (the pinned fp32 chain of down_project, one
    bottleneck shared by all heads): the orientation of h @ W_down (a
    transposed W_down would fail) to within the chain's rounding."""
    _, _, _, h, Wdown, _, _, _ = case(56, B=2, N=30, D=96, dl=24)
    got = oracle.latent_bottleneck(h, Wdown, "f32").astype(np.float64)
    want = h.astype(np.float64) @ Wdown.astype(np.float64)
    np.testing.assert_allclose(got, want, rtol=0, atol=2e-5)
