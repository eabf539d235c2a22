"""Device-side set-up of the DAR workloads: seeded inputs uploaded to the GPU,
caches filled through ``dar_cache_append``, and the algorithmic byte / FLOP
counts the benchmark divides by.  Plumbing only -- no method arithmetic.
"""
from __future__ import annotations

import math

import numpy as np
import torch

from . import dar
from . import inputs as I

TORCH_DTYPE = {"f32": torch.float32, "bf16": torch.bfloat16}
ESIZE = {"f32": 4, "bf16": 2}


def upload(a: np.ndarray, dtype: str, device="cuda") -> torch.Tensor:
    """Storage-type numpy array (float32, or uint16 bf16 bits) -> device tensor."""
    a = np.ascontiguousarray(a)
    if dtype == "bf16":
        return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).to(device)
    return torch.from_numpy(a).to(device)


def download(t: torch.Tensor) -> np.ndarray:
    """Device tensor -> storage-type numpy array (bf16 as uint16 bits)."""
    t = t.detach().to("cpu").contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def to_f64(a: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "bf16":
        return I.bf16_bits_to_f32(a).astype(np.float64)
    return a.astype(np.float64)


# ------------------------------------------------------------------------ decode

def cache_pages_needed(lens, w, extra_tokens=0):
    """Tokens each sequence will hold in pages after ``extra_tokens`` more appends."""
    return np.maximum(np.asarray(lens, dtype=np.int64) + extra_tokens - w, 0)


class DecodeWorkload:
    """A filled mixed-dimension cache for a :class:`inputs.Decode` config.

    The history of every sequence is generated from its seeded stream and
    appended through ``dar_cache_append`` in chunks of ``chunk`` tokens (with
    per-sequence counts for ragged lengths).  ``extra_tokens`` reserves pages
    for later decode steps."""

    def __init__(self, cfg: I.Decode, extra_tokens=0, chunk=4096, device="cuda", keep_history=False,
                 lens=None):
        self.cfg = cfg
        self.device = device
        self.lens = I.decode_lengths(cfg) if lens is None else np.asarray(lens, dtype=np.int64)
        table, num_pages = I.page_assignment(cfg, cache_pages_needed(self.lens, cfg.w, extra_tokens))
        self.table = table
        self.cache = dar.DarCache(cfg.B, cfg.Hkv, cfg.dd, cfg.w, table.shape[1], num_pages,
                                  dtype=TORCH_DTYPE[cfg.dtype], block_table=torch.from_numpy(table),
                                  device=device)
        Dk, Uk, Dv, Uv = I.projections(cfg.seed, cfg.Hkv, cfg.d, cfg.dd)
        self.proj_host = (Dk, Uk, Dv, Uv)
        self.Dk, self.Uk, self.Dv, self.Uv = (upload(x, "f32", device) for x in (Dk, Uk, Dv, Uv))
        self.history = {} if keep_history else None
        Lmax = int(self.lens.max()) if len(self.lens) else 0
        hist = [I.decode_history(cfg, b, int(self.lens[b])) for b in range(cfg.B)]
        if keep_history:
            self.history = hist
        for t0 in range(0, Lmax, chunk):
            n = min(chunk, Lmax - t0)
            kc = np.zeros((cfg.B, cfg.Hkv, n, cfg.d), dtype=hist[0][0].dtype)
            vc = np.zeros_like(kc)
            counts = np.clip(self.lens - t0, 0, n).astype(np.int32)
            for b in range(cfg.B):
                c = int(counts[b])
                if c:
                    kc[b, :, :c] = hist[b][0][:, t0:t0 + c]
                    vc[b, :, :c] = hist[b][1][:, t0:t0 + c]
            dar.dar_cache_append(self.cache, upload(kc, cfg.dtype, device), upload(vc, cfg.dtype, device),
                                 self.Dk, self.Dv, n_per_seq=torch.from_numpy(counts).to(device))
        torch.cuda.synchronize()
        self.q_host = I.decode_query(cfg)
        self.q = upload(self.q_host, cfg.dtype, device)
        self.workspace = dar.decode_workspace(self.cache, cfg.Hq)

    def history_arrays(self):
        """Stacked histories ``[B, Hkv, Lmax, d]`` (zero-padded) for the oracle."""
        cfg = self.cfg
        Lmax = int(self.lens.max())
        dt = self.history[0][0].dtype
        k = np.zeros((cfg.B, cfg.Hkv, Lmax, cfg.d), dtype=dt)
        v = np.zeros_like(k)
        for b, (kb, vb) in enumerate(self.history):
            k[b, :, :kb.shape[1]] = kb
            v[b, :, :vb.shape[1]] = vb
        return k, v

    def decode(self, out=None, stream=None):
        return dar.dar_attn_decode(self.cache, self.q, self.Uk, self.Uv, self.workspace, out=out, stream=stream)


def decode_cache_bytes(cfg: I.Decode, lens) -> int:
    """Cache bytes one decode step must read: per (b, KV head), the ring keys and
    values at d plus the paged keys and values at d_down."""
    e = ESIZE[cfg.dtype]
    lens = np.asarray(lens, dtype=np.int64)
    nwin = np.minimum(lens, cfg.w)
    ndist = lens - nwin
    return int(cfg.Hkv * np.sum(nwin * 2 * cfg.d * e + ndist * 2 * cfg.dd * e))


def decode_step_bytes(cfg: I.Decode, lens) -> int:
    """Algorithmic bytes of one decode attention call: the cache, the queries and the outputs."""
    e = ESIZE[cfg.dtype]
    return decode_cache_bytes(cfg, lens) + 2 * cfg.B * cfg.Hq * cfg.d * e


def append_step_bytes(cfg: I.Decode, lens) -> int:
    """Algorithmic bytes of appending one token per sequence: read the new k, v;
    for sequences past the window read the leaving ring row and write its
    d_down vectors; write the new ring row."""
    e = ESIZE[cfg.dtype]
    lens = np.asarray(lens, dtype=np.int64)
    migrating = int(np.sum(lens + 1 > cfg.w))
    per_head_new = 2 * cfg.d * e * 2               # read k_new, v_new; write ring rows
    per_head_mig = 2 * cfg.d * e + 2 * cfg.dd * e  # read leaving rows; write bottleneck rows
    return cfg.Hkv * (cfg.B * per_head_new + migrating * per_head_mig)


class LatentDecodeWorkload:
    """A filled cache of the latent form for an :class:`inputs.LatentDecode`
    config: every token's hidden state goes through ``dar_latent_append``
    (which computes its bottleneck), in chunks, with per-sequence counts; the
    absorbed maps come from ``dar_latent_absorb``."""

    def __init__(self, cfg: I.LatentDecode, extra_tokens=0, chunk=1024, device="cuda", keep_history=False):
        self.cfg = cfg
        self.lens = I.decode_lengths(cfg)
        cap = self.lens + extra_tokens
        table, num_pages = I.page_assignment(cfg, cap)
        self.cache = dar.DarLatentCache(cfg.B, cfg.Hkv, cfg.D, cfg.dl, cfg.w, table.shape[1], num_pages,
                                        block_table=torch.from_numpy(table), device=device)
        self.proj_host = I.latent_projections(cfg.seed, cfg.Hkv, cfg.D, cfg.dl, cfg.d)
        self.Wdown, Wup, WK, WV = (upload(x, "f32", device) for x in self.proj_host)
        self.A_K, self.A_V = dar.dar_latent_absorb(Wup, WK, WV)
        hist = [I.latent_history(cfg, b, int(self.lens[b])) for b in range(cfg.B)]
        self.history = hist if keep_history else None
        Lmax = int(self.lens.max())
        for t0 in range(0, Lmax, chunk):
            n = min(chunk, Lmax - t0)
            hc = np.zeros((cfg.B, n, cfg.D), dtype=np.uint16)
            kc = np.zeros((cfg.B, cfg.Hkv, n, cfg.d), dtype=np.uint16)
            vc = np.zeros_like(kc)
            counts = np.clip(self.lens - t0, 0, n).astype(np.int32)
            for b in range(cfg.B):
                c = int(counts[b])
                if c:
                    hb, kb, vb = hist[b]
                    hc[b, :c], kc[b, :, :c], vc[b, :, :c] = hb[t0:t0 + c], kb[:, t0:t0 + c], vb[:, t0:t0 + c]
            dar.dar_latent_append(self.cache, upload(hc, "bf16", device), upload(kc, "bf16", device),
                                  upload(vc, "bf16", device), self.Wdown,
                                  n_per_seq=torch.from_numpy(counts).to(device))
        torch.cuda.synchronize()
        self.q_host = I.normal_array(cfg.seed, I.S_QDEC, (cfg.B, cfg.Hq, cfg.d), dtype=cfg.dtype)
        self.q = upload(self.q_host, "bf16", device)
        self.workspace = dar.latent_decode_workspace(self.cache, cfg.Hq)

    def history_arrays(self, seqs):
        """Zero-padded histories of the listed sequences for the oracle:
        ``k, v [n,Hkv,Lmax,d]`` and ``h [n,Lmax,D]``."""
        cfg = self.cfg
        Lm = max(int(self.lens[b]) for b in seqs)
        k = np.zeros((len(seqs), cfg.Hkv, Lm, cfg.d), dtype=np.uint16)
        v = np.zeros_like(k)
        h = np.zeros((len(seqs), Lm, cfg.D), dtype=np.uint16)
        for i, b in enumerate(seqs):
            hb, kb, vb = self.history[b]
            h[i, :hb.shape[0]], k[i, :, :kb.shape[1]], v[i, :, :vb.shape[1]] = hb, kb, vb
        return k, v, h

    def decode(self, out=None, stream=None):
        return dar.dar_latent_decode(self.cache, self.q, self.A_K, self.A_V, self.workspace, out=out, stream=stream)


def latent_decode_bytes(cfg: I.LatentDecode, lens) -> int:
    """Algorithmic bytes of one latent decode call: per sequence the window's
    keys and values per KV head at d, the bottleneck of each distant token once
    (d_lat, shared by every head), and the queries and outputs."""
    e = ESIZE[cfg.dtype]
    lens = np.asarray(lens, dtype=np.int64)
    nwin = np.minimum(lens, cfg.w)
    return int(np.sum(cfg.Hkv * nwin * 2 * cfg.d * e + (lens - nwin) * cfg.dl * e) + 2 * cfg.B * cfg.Hq * cfg.d * e)


# ------------------------------------------------------------------------ prefill

def prefill_pairs(N: int, w: int):
    """(local pairs, global pairs) per head of a causal prefill over N positions."""
    m = min(N, w)
    local = m * (m + 1) // 2 + max(0, N - w) * w  # sum over i of min(i + 1, w)
    glob = N * (N + 1) // 2 - local
    return local, glob


def prefill_flops(cfg: I.Prefill) -> float:
    """Algorithmic FLOPs of the attention contractions: 4d per local pair (q.k and
    p.v), 4 d_down per global pair (q~.k^D and p.v^D), and per query the q Uk^T
    and (o_glob) Uv lifts, 2 * 2 * d * d_down."""
    local, glob = prefill_pairs(cfg.N, cfg.w)
    heads = cfg.B * cfg.Hq
    return float(heads * (local * 4 * cfg.d + glob * 4 * cfg.dd + cfg.N * 4 * cfg.d * cfg.dd))


def prefill_backward_flops(cfg: I.Prefill) -> float:
    """Algorithmic FLOPs of the backward pass: per local pair five d-wide
    contractions (scores recomputed, dP, dq, dk, dv: 10 d), per global pair the
    same five in d_down plus the global value sum the Uv gradient needs
    (12 d_down); per query row q Uk^T, dO Uv^T, the dq lift and the two
    projection-gradient outer products; per key the dk, dv lifts and two more
    outer products (each 2 d d_down)."""
    local, glob = prefill_pairs(cfg.N, cfg.w)
    heads = cfg.B * cfg.Hq
    rows = heads * cfg.N
    keys = cfg.B * cfg.Hkv * cfg.N
    dd2 = 2 * cfg.d * cfg.dd
    return float(heads * (local * 10 * cfg.d + glob * 12 * cfg.dd) + rows * 5 * dd2 + keys * 4 * dd2)


def prefill_exps(cfg: I.Prefill) -> int:
    local, glob = prefill_pairs(cfg.N, cfg.w)
    return cfg.B * cfg.Hq * (local + glob)


class PrefillWorkload:
    def __init__(self, cfg: I.Prefill, device="cuda"):
        self.cfg = cfg
        x = I.prefill_inputs(cfg)
        self.host = x
        self.q, self.k, self.v = (upload(x[n], cfg.dtype, device) for n in ("q", "k", "v"))
        self.Dk, self.Uk, self.Dv, self.Uv = (upload(x[n], "f32", device) for n in ("Dk", "Uk", "Dv", "Uv"))
        self.out = torch.empty_like(self.q)
        nbytes = dar.dar_prefill_workspace_bytes(TORCH_DTYPE[cfg.dtype], cfg.B, cfg.Hkv, cfg.N, cfg.dd)
        self.workspace = torch.empty(max(1, nbytes), dtype=torch.uint8, device=device)

    def run(self, stream=None):
        return dar.dar_attn_prefill(self.q, self.k, self.v, self.Dk, self.Uk, self.Dv, self.Uv, self.cfg.w,
                                    out=self.out, workspace=self.workspace, stream=stream)


def geometric_mean(xs):
    xs = [x for x in xs if x > 0]
    return math.exp(sum(math.log(x) for x in xs) / len(xs)) if xs else 0.0
