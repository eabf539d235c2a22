"""Pins for the backward oracle (oracle.backward, Sec. 2.3 training): each
test checks it against something other than itself -- central finite
differences of the forward oracle (pinned in test_oracle_pins.py), torch's
automatic differentiation of an independently written float64 forward,
torch's scaled_dot_product_attention backward where the method reduces to
standard attention, and exact zeros where a projection cannot influence the
loss."""
import numpy as np
import pytest

import oracle
from paper_2606_18587_gb300 import inputs as I

torch = pytest.importorskip("torch")

NAMES = ("q", "k", "v", "Dk", "Uk", "Dv", "Uv")


def case(seed, B=1, Hq=2, Hkv=1, N=20, d=8, dd=4, dtype="f32"):
    x = dict(q=I.normal_array(seed, I.S_Q, (B, Hq, N, d), dtype=dtype),
             k=I.normal_array(seed, I.S_K, (B, Hkv, N, d), dtype=dtype),
             v=I.normal_array(seed, I.S_V, (B, Hkv, N, d), dtype=dtype))
    x["Dk"], x["Uk"], x["Dv"], x["Uv"] = I.projections(seed, Hkv, d, dd)
    dout = I.normal_array(seed + 1, I.S_Q, (B, Hq, N, d), dtype=dtype)
    return x, dout


def loss(x, dout, w, dtype):
    """sum(dout * o) with o from the forward oracle (float64 from here on)."""
    o = oracle.prefill(x["q"], x["k"], x["v"], x["Dk"], x["Uk"], x["Dv"], x["Uv"], w, dtype, nthreads=1)
    return float(np.sum(oracle.to_f64(dout, dtype) * o))


@pytest.mark.parametrize("w", [0, 3, 7, 20])
def test_backward_matches_finite_differences(w):
    """Every gradient entry equals the central difference of the forward
    oracle's loss.  Steps are powers of two so the perturbed float32 inputs
    are exact; the inputs that reach the loss through the float32 rounding of
    k^D, v^D (k, v, Dk, Dv) take a larger step, so that rounding's noise stays
    below the tolerance."""
    x, dout = case(21 + w, Hq=2, Hkv=1)
    g = oracle.backward(x["q"], x["k"], x["v"], x["Dk"], x["Uk"], x["Dv"], x["Uv"], dout, w, "f32", nthreads=1)
    key = {"q": "dq", "k": "dk", "v": "dv", "Dk": "dDk", "Uk": "dUk", "Dv": "dDv", "Uv": "dUv"}
    for name in NAMES:
        h = 2.0 ** -12 if name in ("q", "Uk", "Uv") else 2.0 ** -7
        rtol = 1e-5 if name in ("q", "Uk", "Uv") else 2e-3
        arr = x[name]
        fd = np.zeros(arr.shape)
        for idx in np.ndindex(arr.shape):
            old = arr[idx]
            arr[idx] = old + np.float32(h)
            lp = loss(x, dout, w, "f32")
            arr[idx] = old - np.float32(h)
            lm = loss(x, dout, w, "f32")
            arr[idx] = old
            fd[idx] = (lp - lm) / (2 * h)
        an = g[key[name]]
        scale = max(1.0, np.abs(fd).max())
        assert np.abs(an - fd).max() <= rtol * scale, (name, np.abs(an - fd).max(), scale)


def torch_forward(t, x, w, dtype, G):
    """An independent float64 forward in torch: k^D, v^D take the stored values
    of Eq. 1 (oracle.down_project, pinned on its own) with the derivative of
    the unrounded product (straight-through), then the explicit lift, the
    Eq. 3 mask and one softmax."""
    q, k, v, Dk, Uk, Dv, Uv = (t[n] for n in NAMES)
    B, Hq, N, d = q.shape

    def stored(prod, name, W):
        val = torch.tensor(oracle.to_f64(oracle.down_project(x[name], x[W], dtype), dtype))
        return prod + (val - prod).detach()

    kd = stored(torch.einsum("bgnt,gtc->bgnc", k, Dk), "k", "Dk")
    vd = stored(torch.einsum("bgnt,gtc->bgnc", v, Dv), "v", "Dv")
    kl = torch.einsum("bgnc,gct->bgnt", kd, Uk)
    vl = torch.einsum("bgnc,gct->bgnt", vd, Uv)
    rep = lambda a: a.repeat_interleave(G, dim=1)
    i = torch.arange(N)[:, None]
    j = torch.arange(N)[None, :]
    local = (i - j) < w
    s_loc = torch.einsum("bhid,bhjd->bhij", q, rep(k)) / np.sqrt(d)
    s_glb = torch.einsum("bhid,bhjd->bhij", q, rep(kl)) / np.sqrt(d)
    s = torch.where(local, s_loc, s_glb).masked_fill(j > i, float("-inf"))
    p = torch.softmax(s, dim=-1)
    return torch.einsum("bhij,bhjd->bhid", torch.where(local, p, 0.0), rep(v)) + \
        torch.einsum("bhij,bhjd->bhid", torch.where(local, 0.0, p), rep(vl))


@pytest.mark.parametrize("dtype,B,Hq,Hkv,N,dd,w", [
    ("f32", 2, 4, 2, 33, 4, 5),
    ("bf16", 1, 4, 1, 40, 8, 9),
    ("bf16", 2, 2, 2, 17, 16, 0),
    ("f32", 1, 3, 3, 25, 16, 25),
])
def test_backward_matches_torch_autograd(dtype, B, Hq, Hkv, N, dd, w):
    """GQA, both storage types, windows from none to everything: every gradient
    equals torch autograd of the independent forward (float64)."""
    x, dout = case(31 + N, B=B, Hq=Hq, Hkv=Hkv, N=N, d=16, dd=dd, dtype=dtype)
    g = oracle.backward(x["q"], x["k"], x["v"], x["Dk"], x["Uk"], x["Dv"], x["Uv"], dout, w, dtype)
    f64 = lambda a, n: torch.tensor(oracle.to_f64(a, dtype) if n in ("q", "k", "v") else a.astype(np.float64),
                                    requires_grad=True)
    t = {n: f64(x[n], n) for n in NAMES}
    o = torch_forward(t, x, w, dtype, Hq // Hkv)
    (o * torch.tensor(oracle.to_f64(dout, dtype))).sum().backward()
    for n, gn in zip(NAMES, ("dq", "dk", "dv", "dDk", "dUk", "dDv", "dUv")):
        ref = t[n].grad.numpy()
        assert np.abs(g[gn] - ref).max() <= 1e-10 * max(1.0, np.abs(ref).max()), (n, np.abs(g[gn] - ref).max())


def test_window_covering_everything_is_standard_attention_backward():
    """w >= N: every pair is local, so dq, dk, dv are the gradients of causal
    attention (torch SDPA, float64) and the projections get exactly zero."""
    x, dout = case(41, B=1, Hq=2, Hkv=2, N=30, d=16, dd=4)
    g = oracle.backward(x["q"], x["k"], x["v"], x["Dk"], x["Uk"], x["Dv"], x["Uv"], dout, 30, "f32")
    q, k, v = (torch.tensor(x[n].astype(np.float64), requires_grad=True) for n in ("q", "k", "v"))
    o = torch.nn.functional.scaled_dot_product_attention(q, k, v, is_causal=True)
    (o * torch.tensor(dout.astype(np.float64))).sum().backward()
    for t, gn in ((q, "dq"), (k, "dk"), (v, "dv")):
        assert np.abs(g[gn] - t.grad.numpy()).max() < 1e-12
    for gn in ("dDk", "dUk", "dDv", "dUv"):
        assert np.all(g[gn] == 0.0)


def test_zero_lift_cuts_the_bottleneck_gradient():
    """Uk = Uv = 0: distant keys and values are the zero vector, so nothing
    reaches Dk, Dv (exact zeros) while Uk and Uv still receive a gradient."""
    x, dout = case(43, N=24, d=8, dd=4)
    x["Uk"][:] = 0
    x["Uv"][:] = 0
    g = oracle.backward(x["q"], x["k"], x["v"], x["Dk"], x["Uk"], x["Dv"], x["Uv"], dout, 4, "f32")
    assert np.all(g["dDk"] == 0.0) and np.all(g["dDv"] == 0.0)
    assert np.abs(g["dUk"]).max() > 1e-3 and np.abs(g["dUv"]).max() > 1e-3
