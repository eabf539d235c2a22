"""GPU cache tests: the Eq. 1 down-projection and the window-exit migration
must be bit-exact against the oracle, and cache indexing must follow the
layout of include/dar.h exactly (ring slot p % w; page block_table[b][p / 64],
row p % 64)."""
import numpy as np
import pytest

import oracle
from paper_2606_18587_gb300 import inputs as I

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("no CUDA device", allow_module_level=True)

from paper_2606_18587_gb300 import dar  # noqa: E402
from paper_2606_18587_gb300 import workloads as W  # noqa: E402


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("dd", [8, 16, 32, 64])
def test_down_project_bit_exact(dtype, dd):
    x = I.normal_array(50 + dd, I.S_K, (2, 3, 300, 64), dtype=dtype)
    Wd = I.normal_array(50 + dd, I.S_DK, (3, 64, dd), std=1 / 8)
    got = W.download(dar.dar_down_project(W.upload(x, dtype), W.upload(Wd, "f32")))
    np.testing.assert_array_equal(got, oracle.down_project(x, Wd, dtype))


def expected_cache(hist, lens, w, dd, Dk, Dv, table, num_pages, dtype):
    """Ring and pool contents implied by the layout, from the oracle's Eq. 1."""
    B = len(hist)
    Hkv = hist[0][0].shape[0]
    dt = hist[0][0].dtype
    ring_k = np.zeros((B, Hkv, w, 64), dtype=dt)
    ring_v = np.zeros_like(ring_k)
    pool_k = np.zeros((max(num_pages, 1), Hkv, 64, dd), dtype=dt)
    pool_v = np.zeros_like(pool_k)
    written = np.zeros(max(num_pages, 1), dtype=bool)
    for b, (kb, vb) in enumerate(hist):
        L = int(lens[b])
        for p in range(max(0, L - w), L):
            ring_k[b, :, p % w] = kb[:, p]
            ring_v[b, :, p % w] = vb[:, p]
        nd = max(0, L - w)
        if nd:
            kd = oracle.down_project(np.ascontiguousarray(kb[None, :, :nd]), Dk, dtype)[0]
            vd = oracle.down_project(np.ascontiguousarray(vb[None, :, :nd]), Dv, dtype)[0]
            for p in range(nd):
                pg = table[b, p // 64]
                pool_k[pg, :, p % 64] = kd[:, p]
                pool_v[pg, :, p % 64] = vd[:, p]
                written[pg] = True
    return ring_k, ring_v, pool_k, pool_v


def check_cache(cache, hist, lens, Dk, Dv, table, dtype):
    rk, rv, pk, pv = expected_cache(hist, lens, cache.w, cache.d_down, Dk, Dv, table, cache.num_pages, dtype)
    np.testing.assert_array_equal(W.download(cache.seq_lens), lens)
    assert cache.device_status() == 0
    # only live slots are defined: slot s of sequence b holds data iff some p < L has p % w == s
    for b in range(len(hist)):
        live = min(int(lens[b]), cache.w)
        np.testing.assert_array_equal(W.download(cache.win_k)[b, :, :live], rk[b, :, :live])
        np.testing.assert_array_equal(W.download(cache.win_v)[b, :, :live], rv[b, :, :live])
        nd = max(0, int(lens[b]) - cache.w)
        gk, gv = W.download(cache.pool_kd), W.download(cache.pool_vd)
        for p in range(nd):
            pg = table[b, p // 64]
            np.testing.assert_array_equal(gk[pg, :, p % 64], pk[pg, :, p % 64])
            np.testing.assert_array_equal(gv[pg, :, p % 64], pv[pg, :, p % 64])


def make(dtype, B, Hkv, dd, w, lens, shuffle, seed):
    cfg = I.Decode("cache-test", seed, B, Hkv, Hkv, 64, dd, w, dtype, L_range=(1, 2), shuffle_pages=shuffle)
    table, npages = I.page_assignment(cfg, W.cache_pages_needed(lens, w))
    cache = dar.DarCache(B, Hkv, dd, w, table.shape[1], npages, dtype=W.TORCH_DTYPE[dtype],
                         block_table=torch.from_numpy(table))
    hist = [I.decode_history(cfg, b, int(lens[b])) for b in range(B)]
    Dk, Uk, Dv, Uv = I.projections(seed, Hkv, 64, dd)
    return cfg, cache, hist, table, Dk, Dv


def append(cache, hist, t0, n, lens, Dk, Dv, dtype):
    B, Hkv = len(hist), hist[0][0].shape[0]
    kc = np.zeros((B, Hkv, n, 64), dtype=hist[0][0].dtype)
    vc = np.zeros_like(kc)
    counts = np.clip(np.asarray(lens) - t0, 0, n).astype(np.int32)
    for b in range(B):
        c = int(counts[b])
        kc[b, :, :c] = hist[b][0][:, t0:t0 + c]
        vc[b, :, :c] = hist[b][1][:, t0:t0 + c]
    dar.dar_cache_append(cache, W.upload(kc, dtype), W.upload(vc, dtype), W.upload(Dk, "f32"),
                         W.upload(Dv, "f32"), n_per_seq=torch.from_numpy(counts).cuda())


@pytest.mark.parametrize("dtype,dd,w,chunk", [
    ("bf16", 16, 5, 1000), ("bf16", 8, 64, 7), ("f32", 32, 3, 2), ("bf16", 64, 100, 1), ("f32", 16, 1, 33),
])
def test_append_matches_layout(dtype, dd, w, chunk):
    """Ragged lengths (0, short, long), appended in chunks smaller and larger
    than the window, pages shuffled: every live ring row and page row is exact."""
    lens = np.array([0, 3, w, w + 1, 150, 333])
    cfg, cache, hist, table, Dk, Dv = make(dtype, len(lens), 2, dd, w, lens, True, 60 + dd + w)
    for t0 in range(0, int(lens.max()), chunk):
        append(cache, hist, t0, min(chunk, int(lens.max()) - t0), lens, Dk, Dv, dtype)
    torch.cuda.synchronize()
    check_cache(cache, hist, lens, Dk, Dv, table, dtype)


def test_token_by_token_equals_bulk():
    lens = np.array([200, 77, 130])
    dtype, dd, w = "bf16", 16, 32
    _, c1, hist, table, Dk, Dv = make(dtype, 3, 2, dd, w, lens, True, 71)
    _, c2, _, _, _, _ = make(dtype, 3, 2, dd, w, lens, True, 71)
    append(c1, hist, 0, int(lens.max()), lens, Dk, Dv, dtype)
    for t in range(int(lens.max())):
        append(c2, hist, t, 1, lens, Dk, Dv, dtype)
    torch.cuda.synchronize()
    for name in ("win_k", "win_v", "pool_kd", "pool_vd", "seq_lens"):
        np.testing.assert_array_equal(W.download(getattr(c1, name)), W.download(getattr(c2, name)))


def test_missing_page_sets_capacity_status():
    lens = np.array([130, 130])
    dtype, dd, w = "bf16", 16, 16
    _, cache, hist, table, Dk, Dv = make(dtype, 2, 1, dd, w, lens, False, 72)
    cache.block_table[1, 1] = -1  # sequence 1 loses its second page
    append(cache, hist, 0, 130, lens, Dk, Dv, dtype)
    torch.cuda.synchronize()
    assert cache.device_status() == dar.DAR_ERR_CAPACITY


def test_append_beyond_capacity_is_refused_on_device():
    lens = np.array([100])
    _, cache, hist, table, Dk, Dv = make("bf16", 1, 1, 16, 8, lens, False, 73)
    before = W.download(cache.pool_kd).copy()
    # capacity is two pages plus the window (136 tokens); 300 do not fit
    k = torch.zeros((1, 1, 300, 64), dtype=torch.bfloat16, device="cuda")
    dar.dar_cache_append(cache, k, k, W.upload(Dk, "f32"), W.upload(Dv, "f32"))
    torch.cuda.synchronize()
    assert cache.device_status() == dar.DAR_ERR_CAPACITY
    assert int(cache.seq_lens.item()) == 0
    np.testing.assert_array_equal(W.download(cache.pool_kd), before)
