"""Host-side model of the decode stream kernel's split-K bookkeeping (no GPU).

The stream kernel lays the stages of every (sequence, KV head, head slice)
group end to end -- ring stages first, then page stages -- and splits them
into ranges: the first Ss stages evenly over the NW warps of the grid
(warp k owns [floor(Ss k / NW), floor(Ss (k + 1) / NW))), the rest into pool
chunks of C stages.  A range cuts groups into parts; the ring and page
segments of a part write records into the range's slots (slot 0 if the
group began before the range, else slot 1), each part adds its stage count
to the group's counter, and the part that completes the count merges the
group by enumerating, for every range the group meets, the records that
range must have written.

This module restates that arithmetic in plain Python and checks the
invariants the kernel relies on, over random batches, lengths, grids and
pool shares:
  * every stage belongs to exactly one range, ranges are contiguous;
  * owner(t) (the range holding stage t) agrees with the range bounds, in
    its exact form and in the kernel's (float estimate, then exact steps);
  * each group's parts add up to its stage count, so exactly one part
    completes it;
  * the records a merge enumerates are exactly the records written;
  * no record slot is written twice for two groups while the first is
    still unmerged;
and checks the kernel's division by the warp count (a float reciprocal with
a one-step correction) exhaustively against integer division.
"""
import random

import numpy as np
import pytest


def stages_of(L, w, tps_w, tps_d):
    """(ring stages, all stages) of one group of a sequence of length L."""
    nwin = min(L, w) if L > 0 else 0
    ndist = L - nwin if L > 0 else 0
    r = -(-nwin // tps_w)
    return r, r + -(-ndist // tps_d)


class Split:
    def __init__(self, S, NW, pool_percent, max_chunks):
        P = S * pool_percent // 100
        self.S, self.NW = S, NW
        self.C = max(1, -(-P // max_chunks))
        self.NC = -(-P // self.C)
        self.Ss = S - P

    def lo(self, k):
        if k <= self.NW:
            return self.Ss * k // self.NW
        return min(self.S, self.Ss + (k - self.NW) * self.C)

    def owner(self, t):
        if t >= self.Ss:
            return self.NW + (t - self.Ss) // self.C
        return ((t + 1) * self.NW - 1) // self.Ss

    def owner_as_kernel(self, t):
        """The kernel's form: a float32 estimate t * (NW / Ss), then exact steps."""
        if t >= self.Ss:
            return self.NW + (t - self.Ss) // self.C
        rate = np.float32(self.NW) / np.float32(self.Ss)
        k = min(self.NW - 1, int(np.float32(t) * rate))
        while k > 0 and self.lo(k) > t:
            k -= 1
        while k + 1 < self.NW and self.lo(k + 1) <= t:
            k += 1
        return k


def simulate(Ls, per_group, NW, w, tps_w, tps_d, pool_percent, max_chunks, rng):
    B = len(Ls)
    st = [stages_of(L, w, tps_w, tps_d) for L in Ls]
    pre = [0]
    for _, n in st:
        pre.append(pre[-1] + n)
    S = pre[B] * per_group
    sp = Split(S, NW, pool_percent, max_chunks)
    nranges = NW + sp.NC
    assert sp.lo(0) == 0 and sp.lo(nranges) == S
    for k in range(nranges):
        assert sp.lo(k) <= sp.lo(k + 1)
    for t in range(S):
        k = sp.owner(t)
        assert sp.lo(k) <= t < sp.lo(k + 1)
        assert sp.owner_as_kernel(t) == k

    written, count, merged, live = {}, {}, set(), {}
    # the warps' own ranges first, then the pool chunks in a random claim order
    order = list(range(NW)) + [NW + u for u in rng.sample(range(sp.NC), sp.NC)]
    for rid in order:
        lo, hi = sp.lo(rid), sp.lo(rid + 1)
        if lo >= hi:
            continue
        b = max(i for i in range(B) if pre[i] * per_group <= lo)
        r, n = st[b]
        gh, j = divmod(lo - pre[b] * per_group, n)
        s = lo
        while s < hi:
            ring = j < r
            G0 = s - j
            G1 = G0 + n
            gid = b * per_group + gh
            slot = 0 if G0 < lo else 1
            if s == hi - 1 or j == n - 1 or j == r - 1:  # segment end: records
                key = (rid, slot, 0 if ring else 1)
                other = live.get(key)
                assert other is None or other == gid or other in merged, (key, other, gid)
                live[key] = gid
                written.setdefault(gid, []).append(key)
            if s == hi - 1 or j == n - 1:  # part end: count
                count[gid] = count.get(gid, 0) + min(hi, G1) - max(lo, G0)
                assert count[gid] <= n
                if count[gid] == n:
                    merged.add(gid)
            s += 1
            if s < hi:
                j += 1
                if j == n:
                    j = 0
                    gh += 1
                    if gh == per_group:
                        gh = 0
                        b += 1
                        while pre[b + 1] == pre[b]:
                            b += 1
                        r, n = st[b]

    for b in range(B):
        r, n = st[b]
        for gh in range(per_group):
            gid = b * per_group + gh
            if n == 0:
                assert gid not in written
                continue
            assert count[gid] == n
            G0 = pre[b] * per_group + gh * n
            G1, GR = G0 + n, G0 + r
            wa, wb = sp.owner(G0), sp.owner(G1 - 1)
            cands = []
            for i in range(2 * (wb - wa + 1)):
                k, typ = wa + i // 2, i % 2
                lo, hi = max(sp.lo(k), G0), min(sp.lo(k + 1), G1)
                has = lo < min(hi, GR) if typ == 0 else max(lo, GR) < hi
                if has:
                    cands.append((k, 0 if G0 < sp.lo(k) else 1, typ))
            assert sorted(cands) == sorted(written[gid]), gid


@pytest.mark.parametrize("seed", range(4))
def test_split_bookkeeping(seed):
    rng = random.Random(seed)
    for _ in range(150):
        B = rng.randint(1, 24)
        Ls = [rng.choice([-1, 0, 1, 31, 32, 33, 128, 129, 300, 1000, rng.randint(0, 3000)]) for _ in range(B)]
        if all(L <= 0 for L in Ls):
            continue
        simulate(Ls, rng.randint(1, 4), rng.choice([8, 37, 64, 152 * 8]), rng.choice([1, 16, 128, 200]),
                 rng.choice([16, 32]), rng.choice([16, 32, 64, 128, 256]), rng.choice([0, 0, 15, 50, 100]),
                 rng.choice([7, 100, 2 * 160 * 8]), rng)


def test_decode160m_split():
    """The benchmark's shape: 32 sequences of 4097 tokens, 12 groups each, 1216 warps."""
    simulate([4097] * 32, 12, 152 * 8, 128, 32, 128, 0, 2 * 160 * 8, random.Random(0))


def test_division_by_warp_count():
    """floor(x / NW) as the kernel computes it (float32 product with 1/NW,
    truncation, one correction each way) for every grid it can launch
    (NW = 8 x CTAs, CTAs <= 160) and every x < NW^2 it is used on."""
    for NW in range(8, 1281, 8):
        inv = np.float32(1.0) / np.float32(NW)
        x = np.arange(NW * NW, dtype=np.int64)
        q = (x.astype(np.float32) * inv).astype(np.int64)
        q = q + ((q + 1) * NW <= x)
        q = q - (q * NW > x)
        assert np.array_equal(q, x // NW), NW
