"""Seeded synthetic inputs shaped like the SENSE workloads.

This module only draws random inputs; it holds no step of the method.  Both
the CUDA path and the CPU oracle receive the same tensors from here.

Recipes (all seeded; per-chunk seeds make large stores reproducible chunk by
chunk, independent of the device that draws them):

* keys: ``n_clusters`` centroids uniform on the unit sphere; each key picks a
  centroid uniformly and adds Gaussian noise, then is put back on the unit
  sphere and stored as bf16.  Noise reading "A" draws N(0, sigma^2/d) per
  coordinate (noise vector norm ~ sigma); reading "B" draws N(0, sigma^2)
  per coordinate.
* subspace keys (approximate-retrieval studies): the clusters and the spread
  within them live in a random ``rank``-dimensional subspace of R^d whose
  coordinates have a power-law spectrum (scale (i+1)^-decay), plus a small
  isotropic noise of norm ~``iso``; back on the unit sphere, bf16.  Hidden
  states concentrate their energy in few directions like this; isotropic
  clusters in d dimensions do not.
* queries: a uniformly chosen key plus Gaussian noise (same readings), back
  on the unit sphere, as bf16; the source key index is returned.
* lattice keys/queries: entries from {-3..3} * 2^-6 (exact in bf16, and all
  dot products are exact in fp32), used to make ties frequent.
* spans: int32 token ids, uniform in [0, vocab) or Zipf(s) by rank
  (P(r) proportional to (r+1)^-s), drawn by inverse CDF.
* gate inputs: fp32 logits N(0, std^2) per tree node row, bf16 hidden states
  N(0, 1); ``plant_gate_rows`` raises chosen child tokens in their parent's
  row so that exact-match and top-k paths are exercised.
"""
from __future__ import annotations

import torch

CHUNK_ROWS = 65536


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) & ((1 << 63) - 1))
    return g


def _sub_seed(seed: int, stream: int, chunk: int = 0) -> int:
    return (int(seed) * 1000003 + stream * 7919 + chunk * 104729) & ((1 << 62) - 1)


def _unit_rows(x: torch.Tensor) -> torch.Tensor:
    # Put draws on the unit sphere (this shapes the input distribution).
    return x / x.norm(dim=1, keepdim=True).clamp_min(1e-30)


def centroids(n_clusters: int, d: int, seed: int = 0, device="cpu") -> torch.Tensor:
    g = _gen(device, _sub_seed(seed, 1))
    c = torch.randn(n_clusters, d, generator=g, device=device, dtype=torch.float32)
    return _unit_rows(c)


def clustered_unit_keys(n: int, d: int, n_clusters: int, sigma: float = 0.3,
                        seed: int = 0, device="cpu", reading: str = "A",
                        out: torch.Tensor | None = None, return_assign: bool = False):
    """bf16 [n, d] keys drawn around ``n_clusters`` unit centroids (and, with
    ``return_assign``, the int32 [n] cluster of each key)."""
    c = centroids(n_clusters, d, seed, device)
    if out is None:
        out = torch.empty(n, d, dtype=torch.bfloat16, device=device)
    assign = torch.empty(n, dtype=torch.int32, device=device) if return_assign else None
    for ci, lo in enumerate(range(0, n, CHUNK_ROWS)):
        hi = min(n, lo + CHUNK_ROWS)
        rows, a = _key_chunk(c, ci, hi - lo, sigma, seed, reading)
        out[lo:hi] = rows
        if assign is not None:
            assign[lo:hi] = a.to(torch.int32)
        del rows
    return (out, assign) if return_assign else out


def _key_chunk(c: torch.Tensor, ci: int, rows: int, sigma: float, seed: int, reading: str):
    """Chunk ``ci`` of a clustered store: (bf16 [rows, d] keys, cluster ids)."""
    n_clusters, d = c.shape
    scale = sigma / (d ** 0.5) if reading == "A" else sigma
    g = _gen(c.device, _sub_seed(seed, 2, ci))
    a = torch.randint(0, n_clusters, (rows,), generator=g, device=c.device)
    e = torch.randn(rows, d, generator=g, device=c.device, dtype=torch.float32)
    x = c[a] + scale * e
    return _unit_rows(x).to(torch.bfloat16), a


class ClusteredStoreRows:
    """Rows of the store ``clustered_unit_keys`` draws, produced chunk by
    chunk on demand (the same values on the same device), for consumers that
    cannot hold the whole store."""

    def __init__(self, n: int, d: int, n_clusters: int, sigma: float = 0.3, seed: int = 0,
                 device="cpu", reading: str = "A"):
        self.n, self.d, self.sigma, self.seed, self.reading = n, d, sigma, seed, reading
        self.c = centroids(n_clusters, d, seed, device)

    def chunk(self, ci: int) -> torch.Tensor:
        lo = ci * CHUNK_ROWS
        hi = min(self.n, lo + CHUNK_ROWS)
        return _key_chunk(self.c, ci, hi - lo, self.sigma, self.seed, self.reading)[0]

    def rows(self, idx: torch.Tensor) -> torch.Tensor:
        """bf16 [len(idx), d]: the store rows at the given indices."""
        idx = idx.to(self.c.device)
        out = torch.empty(idx.shape[0], self.d, dtype=torch.bfloat16, device=self.c.device)
        chunks = torch.div(idx, CHUNK_ROWS, rounding_mode="floor")
        for ci in sorted(set(chunks.tolist())):
            sel = chunks == ci
            out[sel] = self.chunk(ci)[idx[sel] - ci * CHUNK_ROWS]
        return out


def noisy_queries(keys, q: int, noise: float = 0.05, seed: int = 0,
                  reading: str = "A"):
    """(bf16 [q, d] queries, int64 [q] source key index).  ``keys`` is the
    store tensor, or a ``ClusteredStoreRows`` for a store that is not held."""
    if isinstance(keys, ClusteredStoreRows):
        n, d, dev, fetch = keys.n, keys.d, keys.c.device, keys.rows
    else:
        n, d = keys.shape
        dev = keys.device
        fetch = lambda s: keys[s]  # noqa: E731
    g = _gen(dev, _sub_seed(seed, 3))
    src = torch.randint(0, n, (q,), generator=g, device=dev)
    scale = noise / (d ** 0.5) if reading == "A" else noise
    e = torch.randn(q, d, generator=g, device=dev, dtype=torch.float32)
    x = fetch(src).float() + scale * e
    return _unit_rows(x).to(torch.bfloat16), src


def subspace_unit_keys(n: int, d: int, n_clusters: int, rank: int = 256, decay: float = 1.0,
                       sigma: float = 0.3, iso: float = 0.05, seed: int = 0, device="cpu",
                       out: torch.Tensor | None = None, return_assign: bool = False):
    """bf16 [n, d] unit keys whose clusters and within-cluster spread lie in a
    random ``rank``-dimensional subspace (power-law coordinate scales), plus
    isotropic noise of norm ~``iso`` (and, with ``return_assign``, the int32
    cluster of each key)."""
    g = _gen(device, _sub_seed(seed, 13))
    # the orthonormal basis is factored on the host in fp64 (no device linear-algebra
    # library needed; the same basis on every machine up to fp64 rounding)
    draw = torch.randn(d, rank, generator=g, device=device)
    basis = torch.linalg.qr(draw.double().cpu())[0].float().to(device)  # [d, rank]
    scale = torch.arange(1, rank + 1, device=device, dtype=torch.float32).pow(-decay)
    scale = scale / scale.norm()
    cz = torch.randn(n_clusters, rank, generator=g, device=device) * scale
    if out is None:
        out = torch.empty(n, d, dtype=torch.bfloat16, device=device)
    assign = torch.empty(n, dtype=torch.int32, device=device) if return_assign else None
    for ci, lo in enumerate(range(0, n, CHUNK_ROWS)):
        hi = min(n, lo + CHUNK_ROWS)
        gc = _gen(device, _sub_seed(seed, 14, ci))
        a = torch.randint(0, n_clusters, (hi - lo,), generator=gc, device=device)
        z = cz[a] + sigma * scale * torch.randn(hi - lo, rank, generator=gc, device=device)
        x = z @ basis.T + (iso / d ** 0.5) * torch.randn(hi - lo, d, generator=gc, device=device)
        out[lo:hi] = _unit_rows(x).to(torch.bfloat16)
        if assign is not None:
            assign[lo:hi] = a.to(torch.int32)
        del z, x
    return (out, assign) if return_assign else out


def lattice_rows(n: int, d: int, seed: int = 0, device="cpu") -> torch.Tensor:
    """bf16 [n, d] with entries in {-3..3} * 2^-6 (exact in bf16)."""
    out = torch.empty(n, d, dtype=torch.bfloat16, device=device)
    for ci, lo in enumerate(range(0, n, CHUNK_ROWS)):
        hi = min(n, lo + CHUNK_ROWS)
        g = _gen(device, _sub_seed(seed, 4, ci))
        v = torch.randint(-3, 4, (hi - lo, d), generator=g, device=device)
        out[lo:hi] = (v.float() * (2.0 ** -6)).to(torch.bfloat16)
    return out


def gaussian_rows_f32(n: int, d: int, seed: int = 0, device="cpu",
                      std: float = 1.0) -> torch.Tensor:
    g = _gen(device, _sub_seed(seed, 5))
    return std * torch.randn(n, d, generator=g, device=device, dtype=torch.float32)


def spans_uniform(n: int, m: int, vocab: int, seed: int = 0, device="cpu") -> torch.Tensor:
    out = torch.empty(n, m, dtype=torch.int32, device=device)
    for ci, lo in enumerate(range(0, n, CHUNK_ROWS * 16)):
        hi = min(n, lo + CHUNK_ROWS * 16)
        g = _gen(device, _sub_seed(seed, 6, ci))
        out[lo:hi] = torch.randint(0, vocab, (hi - lo, m), generator=g, device=device,
                                   dtype=torch.int32)
    return out


def zipf_cdf(vocab: int, s: float = 1.1, device="cpu") -> torch.Tensor:
    r = torch.arange(1, vocab + 1, dtype=torch.float64, device=device)
    w = r.pow(-s)
    c = torch.cumsum(w, 0)
    return c / c[-1]


def spans_zipf(n: int, m: int, vocab: int, s: float = 1.1, seed: int = 0,
               device="cpu") -> torch.Tensor:
    """int32 [n, m] token ids; token id = frequency rank, P(r) ~ (r+1)^-s."""
    cdf = zipf_cdf(vocab, s, device)
    out = torch.empty(n, m, dtype=torch.int32, device=device)
    for ci, lo in enumerate(range(0, n, CHUNK_ROWS * 16)):
        hi = min(n, lo + CHUNK_ROWS * 16)
        g = _gen(device, _sub_seed(seed, 7, ci))
        u = torch.rand(hi - lo, m, generator=g, device=device, dtype=torch.float64)
        t = torch.searchsorted(cdf, u.reshape(-1), right=True).clamp_max(vocab - 1)
        out[lo:hi] = t.reshape(hi - lo, m).to(torch.int32)
    return out



def spans_cluster_template(assign: torch.Tensor, n_clusters: int, m: int, vocab: int,
                           s: float = 1.1, seed: int = 0) -> torch.Tensor:
    """int32 [n, m] spans that share prefixes within a key cluster.

    Each cluster owns one Zipf(s) template span; a key of that cluster keeps
    the template's first l tokens, l uniform on {0..m}, and draws the rest
    from Zipf(s) (nearby hidden states tend to continue alike)."""
    dev = assign.device
    n = assign.shape[0]
    tmpl = spans_zipf(n_clusters, m, vocab, s, seed=_sub_seed(seed, 10), device=dev)
    fresh = spans_zipf(n, m, vocab, s, seed=_sub_seed(seed, 11), device=dev)
    out = torch.empty(n, m, dtype=torch.int32, device=dev)
    col = torch.arange(m, device=dev)
    for ci, lo in enumerate(range(0, n, CHUNK_ROWS * 16)):
        hi = min(n, lo + CHUNK_ROWS * 16)
        g = _gen(dev, _sub_seed(seed, 12, ci))
        keep = torch.randint(0, m + 1, (hi - lo, 1), generator=g, device=dev)
        a = assign[lo:hi].long()
        out[lo:hi] = torch.where(col[None, :] < keep, tmpl[a], fresh[lo:hi])
    return out

def gate_logits(q: int, rows: int, vocab: int, std: float = 3.0, seed: int = 0,
                device="cpu", out: torch.Tensor | None = None) -> torch.Tensor:
    """fp32 [q, rows, vocab] i.i.d. N(0, std^2)."""
    if out is None:
        out = torch.empty(q, rows, vocab, dtype=torch.float32, device=device)
    for qi in range(q):
        g = _gen(device, _sub_seed(seed, 8, qi))
        out[qi].normal_(0.0, std, generator=g)
    return out


def gate_hidden(q: int, rows: int, d: int, seed: int = 0, device="cpu") -> torch.Tensor:
    g = _gen(device, _sub_seed(seed, 9))
    return torch.randn(q, rows, d, generator=g, device=device,
                       dtype=torch.float32).to(torch.bfloat16)


def plant_gate_rows(root_logits: torch.Tensor, node_logits: torch.Tensor,
                    tokens: torch.Tensor, parent: torch.Tensor,
                    num_nodes: torch.Tensor, seed: int = 0,
                    p_top: float = 0.6, p_near: float = 0.15,
                    p_sharp: float = 0.2) -> None:
    """In-place structure for gate tests (CPU tensors).

    For each tree node n, the row that predicts it is its parent's row (the
    root row for depth 0).  A seeded fraction ``p_top`` of nodes gets +20 on
    its token in that row (usually the argmax afterwards), ``p_near`` gets
    its token set just below the row maximum (a near-top alternative), and a
    fraction ``p_sharp`` of all rows is multiplied by 10 (low entropy).
    """
    g = _gen("cpu", _sub_seed(seed, 10))
    qn, cap, _ = node_logits.shape
    for q in range(qn):
        nn = int(num_nodes[q])
        u = torch.rand(nn, generator=g, dtype=torch.float64)
        for n in range(nn):
            p = int(parent[q, n])
            row = root_logits[q] if p < 0 else node_logits[q, p]
            t = int(tokens[q, n])
            if u[n] < p_top:
                row[t] += 20.0
            elif u[n] < p_top + p_near:
                row[t] = row.max() - 0.05 - 0.5 * float(torch.rand(1, generator=g))
        sharp = torch.rand(cap + 1, generator=g) < p_sharp
        if sharp[0]:
            root_logits[q] *= 10.0
        for n in range(nn):
            if sharp[n + 1]:
                node_logits[q, n] *= 10.0
