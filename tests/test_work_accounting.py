"""The benchmark's algorithmic-work counts, which every roofline fraction
divides by, against brute-force enumeration on small shapes: the causal
(i, j) pairs split by Eq. 3 (local iff i - j < w), the exponentials, the
FLOPs of the forward and the backward, and the cache bytes a decode step or
a latent-form decode step must read."""
import itertools

import numpy as np
import pytest

pytest.importorskip("torch")

from paper_2606_18587_gb300 import inputs as I  # noqa: E402
from paper_2606_18587_gb300 import workloads as W  # noqa: E402


def pairs_brute(N, w):
    loc = glob = 0
    for i in range(N):
        for j in range(i + 1):
            if i - j < w:
                loc += 1
            else:
                glob += 1
    return loc, glob


@pytest.mark.parametrize("N,w", [(1, 1), (7, 0), (7, 3), (40, 40), (40, 100), (65, 17), (130, 64)])
def test_prefill_pairs(N, w):
    assert W.prefill_pairs(N, w) == pairs_brute(N, w)


@pytest.mark.parametrize("B,Hq,Hkv,N,dd,w", [(1, 2, 1, 33, 8, 5), (2, 4, 2, 20, 16, 0), (1, 3, 3, 17, 64, 40)])
def test_prefill_flops_and_exps(B, Hq, Hkv, N, dd, w):
    cfg = I.Prefill("acct", 1, B, Hq, Hkv, N, 64, dd, w, "bf16")
    loc, glob = pairs_brute(N, w)
    heads, d = B * Hq, 64
    # forward: q.k and p.v per pair (2 FLOP per multiply-add), plus the q Uk^T and (o_glob) Uv lifts per row
    fwd = heads * (loc * 2 * 2 * d + glob * 2 * 2 * dd + N * 2 * (2 * d * dd))
    assert W.prefill_flops(cfg) == fwd
    assert W.prefill_exps(cfg) == heads * (loc + glob)
    # backward: five contractions per pair (scores, dP, dq, dk, dv), the global
    # value sum O^D beside them; per row the two lifts in, the dq lift and two
    # outer products; per key the dk, dv lifts and two outer products
    bwd = heads * (loc * 5 * 2 * d + glob * 6 * 2 * dd) + heads * N * 5 * (2 * d * dd) + \
        B * Hkv * N * 4 * (2 * d * dd)
    assert W.prefill_backward_flops(cfg) == bwd


def test_decode_bytes_per_token():
    """Per (sequence, KV head): every window token's key and value at d, every
    distant token's bottleneck key and value at d_down (bf16), plus q and o."""
    cfg = I.Decode("acct", 1, 3, 4, 2, 64, 16, 10, "bf16", L=1)
    lens = np.array([0, 7, 25])
    want = 0
    for b, L in enumerate(lens):
        for g, j in itertools.product(range(cfg.Hkv), range(L)):
            want += 2 * 64 * 2 if L - 1 - j < cfg.w else 2 * 16 * 2
    assert W.decode_cache_bytes(cfg, lens) == want
    assert W.decode_step_bytes(cfg, lens) == want + 2 * cfg.B * cfg.Hq * 64 * 2


def test_latent_decode_bytes_per_token():
    """Window tokens: key and value per KV head at d; distant tokens: one
    d_lat bottleneck for all heads (bf16); plus q and o."""
    cfg = I.LatentDecode("acct", 1, 3, 8, 2, 64, 96, 64, 10, L=1)
    lens = np.array([0, 9, 40])
    want = 0
    for L in lens:
        for j in range(L):
            want += cfg.Hkv * 2 * 64 * 2 if L - 1 - j < cfg.w else cfg.dl * 2
    assert W.latent_decode_bytes(cfg, lens) == want + 2 * cfg.B * cfg.Hq * 64 * 2


def test_append_step_bytes():
    """One token per sequence: read its key and value, write them to the ring;
    when the sequence is past the window, read the leaving ring row and write
    its two bottleneck vectors (bf16)."""
    cfg = I.Decode("acct", 1, 4, 4, 2, 64, 16, 8, "bf16", L=1)
    lens = np.array([0, 7, 8, 30])  # lengths before the append
    want = 0
    for L in lens:
        for g in range(cfg.Hkv):
            want += 2 * 64 * 2 * 2  # read k_new, v_new; write the ring rows
            if L + 1 > cfg.w:  # position L - w + 1 leaves the window
                want += 2 * 64 * 2 + 2 * 16 * 2
    assert W.append_step_bytes(cfg, lens) == want
