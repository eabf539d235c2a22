"""Pins for the oracle of Sec. 5's direct lower-dimensional global attention
(oracle.attention_rows_direct / prefill_direct / decode_direct): each test
checks it against something other than itself -- the standard DAR oracle
(pinned in test_oracle_pins.py) through the absorption identity of Eq. 2,
torch's scaled_dot_product_attention in float64, and invariants of Eq. 3."""
import numpy as np
import pytest

import oracle
from paper_2606_18587_gb300 import inputs as I

torch = pytest.importorskip("torch")


def case(seed, B=2, Hq=4, Hkv=2, N=40, d=16, dd=4, dtype="f32"):
    q = I.normal_array(seed, I.S_Q, (B, Hq, N, d), dtype=dtype)
    k = I.normal_array(seed, I.S_K, (B, Hkv, N, d), dtype=dtype)
    v = I.normal_array(seed, I.S_V, (B, Hkv, N, d), dtype=dtype)
    Dk, Uk, Dv, Uv = I.projections(seed, Hkv, d, dd)
    qd = I.normal_array(seed + 7, I.S_Q, (B, Hq, N, dd), dtype=dtype)
    return q, qd, k, v, Dk, Uk, Dv, Uv


def sdpa(q, k, v, scale):
    """Causal attention of one head with torch (float64, CPU)."""
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a))[None, None]
    return torch.nn.functional.scaled_dot_product_attention(t(q), t(k), t(v), is_causal=True,
                                                            scale=scale)[0, 0].numpy()


@pytest.mark.parametrize("w", [0, 1, 7, 16, 39, 64])
def test_absorbed_queries_reduce_to_standard_dar(w):
    """With q^D = (scale / scale_down) q Uk^T and Wo = Uv the direct variant is
    the standard method in its absorbed form (Eq. 2 by linearity): equal up to
    the float32 rounding of q^D."""
    q, _, k, v, Dk, Uk, Dv, Uv = case(11)
    d, dd = q.shape[3], Uk.shape[1]
    scale, scale_down = 1 / np.sqrt(d), 1 / np.sqrt(dd)
    G = q.shape[1] // k.shape[1]
    qd = np.empty(q.shape[:3] + (dd,), dtype=np.float32)
    for h in range(q.shape[1]):
        qd[:, h] = (q[:, h].astype(np.float64) @ Uk[h // G].astype(np.float64).T * (scale / scale_down)).astype(np.float32)
    want = oracle.prefill(q, k, v, Dk, Uk, Dv, Uv, w, "f32", scale=scale)
    got = oracle.prefill_direct(q, qd, k, v, Dk, Dv, Uv, w, "f32", scale=scale, scale_down=scale_down)
    assert np.abs(got - want).max() < 2e-5


def test_window_covering_everything_is_causal_attention():
    """w >= N: every pair is local, so q^D, the d_down cache and Wo play no part."""
    q, qd, k, v, Dk, _, Dv, Uv = case(12)
    N, d = q.shape[2], q.shape[3]
    got = oracle.prefill_direct(q, qd, k, v, Dk, Dv, Uv, N, "f32")
    G = q.shape[1] // k.shape[1]
    for b in range(q.shape[0]):
        for h in range(q.shape[1]):
            want = sdpa(q[b, h].astype(np.float64), k[b, h // G].astype(np.float64), v[b, h // G].astype(np.float64),
                        1 / np.sqrt(d))
            assert np.abs(got[b, h] - want).max() < 1e-12


def test_zero_window_is_attention_in_d_down():
    """w = 0: every pair is global, so each row is causal attention of q^D over
    the d_down keys with the mapped values v^D Wo (Eq. 1 for k^D, v^D)."""
    q, qd, k, v, Dk, _, Dv, Wo = case(13, dd=8)
    dd = qd.shape[3]
    got = oracle.prefill_direct(q, qd, k, v, Dk, Dv, Wo, 0, "f32")
    kd = oracle.to_f64(oracle.down_project(k, Dk, "f32"), "f32")
    vd = oracle.to_f64(oracle.down_project(v, Dv, "f32"), "f32")
    G = q.shape[1] // k.shape[1]
    for b in range(q.shape[0]):
        for h in range(q.shape[1]):
            g = h // G
            want = sdpa(qd[b, h].astype(np.float64), kd[b, g], vd[b, g] @ Wo[g].astype(np.float64), 1 / np.sqrt(dd))
            assert np.abs(got[b, h] - want).max() < 1e-12


def test_local_rows_ignore_the_global_path():
    """Rows i < w see only local keys (Eq. 3): changing q^D or Wo leaves them
    bit-identical, while rows past the window change."""
    q, qd, k, v, Dk, _, Dv, Wo = case(14)
    w = 10
    a = oracle.prefill_direct(q, qd, k, v, Dk, Dv, Wo, w, "f32")
    b = oracle.prefill_direct(q, -qd, k, v, Dk, Dv, 2 * Wo, w, "f32")
    assert np.array_equal(a[:, :, :w], b[:, :, :w])
    assert np.abs(a[:, :, w:] - b[:, :, w:]).max() > 1e-3


def test_decode_is_the_last_prefill_row():
    """A decode step at position L-1 equals row L-1 of the forward (bf16)."""
    q, qd, k, v, Dk, _, Dv, Wo = case(15, B=2, N=33, dtype="bf16")
    lens = [33, 20]
    q_last = np.stack([q[b, :, lens[b] - 1] for b in range(2)])
    qd_last = np.stack([qd[b, :, lens[b] - 1] for b in range(2)])
    got = oracle.decode_direct(q_last, qd_last, k, v, lens, Dk, Dv, Wo, 8, "bf16")
    for b in range(2):
        L = lens[b]
        full = oracle.prefill_direct(np.ascontiguousarray(q[b:b + 1, :, :L]), np.ascontiguousarray(qd[b:b + 1, :, :L]),
                                     np.ascontiguousarray(k[b:b + 1, :, :L]), np.ascontiguousarray(v[b:b + 1, :, :L]),
                                     Dk, Dv, Wo, 8, "bf16")
        assert np.array_equal(got[b], full[0, :, L - 1])
