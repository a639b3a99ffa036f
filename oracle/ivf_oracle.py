"""Plain CPU oracle of the approximate retrieval path (test infrastructure only).

Only the test suite, the smoke check and the CPU legs of the benchmark import
this module; the product library never uses it and shares no code with it.

SENSE retrieves with an approximate nearest-neighbour index over projected
keys (Sec. 3.2.2 Eq. 7, ANN(k_t, C_db, N')).  App. E fixes the setup: final
layer hidden states are projected by PCA to 64 dimensions and L2-normalised
(Alg. 2, query construction k = L2Norm(PCA(h))), and a FAISS IVF-PQ index
with nlist = 4096 Voronoi cells, nprobe = 32 probed cells and pq_m = 16
sub-quantizers answers the top-N' query.  The functions below restate that
pipeline in numpy:

  project        k = L2Norm(W (h - mu)) for a PCA basis W [v, d]
  kmeans         Lloyd iterations (coarse quantizer and PQ codebooks)
  ivf_build      cell assignment, inverted lists, flat vectors or PQ codes
  ivf_search     coarse top-nprobe, list scan, exact top-k of the
                 approximate scores
  rescore_topk   Eq. 8's sim(h, k_i) over the N' retrieved candidates,
                 exactly, and the top N of them

Precision.  The projection (query and key construction) is a plain linear
map followed by a normalisation, and its oracle is that definition in fp64:
y = (x - mu) W^T summed exactly in fp64 over the hidden size, then y / ||y||.
The CUDA path computes it in fp32; the tests compare the two within an
error bound derived from the fp32 arithmetic, not bit for bit.

Every later step ends in an integer decision (a cell, a code, a probe set, a
top-k index).  FAISS takes those decisions in fp32, and so does this oracle,
on vectors it is given (the tests hand both sides the same projected
vectors): dot products and squared distances in the projected space
(dimension <= 128) are the plain left-to-right sums, each product rounded
to fp32 before it is added (no fused multiply-add; ``dot_seq``, ``l2_seq``).
k-means means are accumulated in 2^-31 fixed point (integer sums do not
depend on the order of the members) and divided in fp64.  The left-to-right
fp32 sum and the fixed-point mean are readings: the paper does not state an
evaluation order.  Pins in tests/test_oracle_ivf.py compare every function
against exact arithmetic, brute force and special cases.
"""
from __future__ import annotations

import numpy as np

from .sense_oracle import bf16_bits_to_f64, scores

F32 = np.float32
FIX = float(2 ** 31)  # fixed-point scale of the k-means sums


# ----------------------------------------------------------------------------
# fp32 reductions in a fixed order
# ----------------------------------------------------------------------------


def dot_seq(a: np.ndarray, b: np.ndarray) -> np.ndarray:
    """sum_j a[..., j] * b[..., j] in fp32, j ascending, products rounded."""
    a = np.asarray(a, dtype=F32)
    b = np.asarray(b, dtype=F32)
    shape = np.broadcast_shapes(a.shape[:-1], b.shape[:-1])
    acc = np.zeros(shape, dtype=F32)
    for j in range(a.shape[-1]):
        acc = (acc + (a[..., j] * b[..., j])).astype(F32)
    return acc


def l2_seq(a: np.ndarray, b: np.ndarray) -> np.ndarray:
    """sum_j (a[..., j] - b[..., j])^2 in fp32, j ascending, no fusion."""
    a = np.asarray(a, dtype=F32)
    b = np.asarray(b, dtype=F32)
    shape = np.broadcast_shapes(a.shape[:-1], b.shape[:-1])
    acc = np.zeros(shape, dtype=F32)
    for j in range(a.shape[-1]):
        t = (a[..., j] - b[..., j]).astype(F32)
        acc = (acc + (t * t)).astype(F32)
    return acc


def _l2_normalize(y: np.ndarray) -> np.ndarray:
    """y / ||y|| per row in fp32 (zero rows stay zero)."""
    nrm = np.sqrt(dot_seq(y, y)).astype(F32)
    out = np.zeros_like(y, dtype=F32)
    nz = nrm > 0
    out[nz] = (y[nz] / nrm[nz, None]).astype(F32)
    return out


# ----------------------------------------------------------------------------
# query / key construction: k = L2Norm(PCA(h))  (Alg. 2; App. E)
# ----------------------------------------------------------------------------


def project(x_bits: np.ndarray, basis: np.ndarray, mean=None, normalize: bool = True):
    """PCA projection of bf16 hidden states, then (optionally) unit L2 norm,
    in fp64 (App. E: PCA to v dimensions, then L2Norm; Alg. 2 builds the
    query as k = L2Norm(PCA(h))).

    x_bits [n, d] uint16 (bf16), basis [v, d] (row o = principal axis o),
    mean [d] or None.  The PCA coordinates are y[i, o] = sum_j (x[i, j] -
    mean[j]) * basis[o, j]; with ``normalize``, y[i] / ||y[i]|| (a zero row
    stays zero).  Returns float64 [n, v].
    """
    x = bf16_bits_to_f64(np.asarray(x_bits))  # exact
    w = np.asarray(basis, dtype=np.float64)
    if mean is not None:
        x = x - np.asarray(mean, dtype=np.float64)[None, :]
    y = x @ w.T
    if not normalize:
        return y
    nrm = np.sqrt((y * y).sum(axis=1))
    out = np.zeros_like(y)
    nz = nrm > 0
    out[nz] = y[nz] / nrm[nz, None]
    return out


# ----------------------------------------------------------------------------
# k-means (the coarse quantizer and the PQ codebooks of the IVF-PQ index)
# ----------------------------------------------------------------------------


def assign_ip(x: np.ndarray, c: np.ndarray) -> np.ndarray:
    """Index of the largest inner product per row (ties: lowest index)."""
    s = dot_seq(np.asarray(x, F32)[:, None, :], np.asarray(c, F32)[None, :, :])
    return np.argmax(s, axis=1).astype(np.int32)  # argmax takes the first maximum


def assign_l2(x: np.ndarray, c: np.ndarray) -> np.ndarray:
    """Index of the nearest centroid in L2 per row (ties: lowest index)."""
    dist = l2_seq(np.asarray(x, F32)[:, None, :], np.asarray(c, F32)[None, :, :])
    return np.argmin(dist, axis=1).astype(np.int32)


def kmeans_update(x: np.ndarray, assign: np.ndarray, prev: np.ndarray, spherical: bool):
    """New centroids: member means (2^-31 fixed point sums, fp64 division,
    rounded to fp32); an empty cluster keeps its previous centroid;
    spherical k-means then puts every centroid on the unit sphere."""
    x = np.asarray(x, F32)
    k, dim = prev.shape
    fx = np.rint(x.astype(np.float64) * FIX).astype(np.int64)
    sums = np.zeros((k, dim), dtype=np.int64)
    np.add.at(sums, assign, fx)
    cnt = np.bincount(assign, minlength=k)
    out = np.array(prev, dtype=F32, copy=True)
    nz = cnt > 0
    out[nz] = ((sums[nz].astype(np.float64) / cnt[nz, None].astype(np.float64))
               * (1.0 / FIX)).astype(F32)
    if spherical:
        out = _l2_normalize(out)
    return out, cnt


def kmeans(x: np.ndarray, init: np.ndarray, iters: int, spherical: bool):
    """Lloyd's algorithm from ``init``: ``iters`` rounds of (assign, update).
    Spherical: inner-product assignment and unit centroids; otherwise L2.
    Returns (centroids [k, dim] f32, assignment of the last round)."""
    c = np.array(init, dtype=F32, copy=True)
    if spherical:
        c = _l2_normalize(c)
    a = np.zeros(len(x), np.int32)
    for _ in range(iters):
        a = assign_ip(x, c) if spherical else assign_l2(x, c)
        c, _ = kmeans_update(x, a, c, spherical)
    return c, a


# ----------------------------------------------------------------------------
# IVF index (App. E: nlist cells, pq_m sub-quantizers)
# ----------------------------------------------------------------------------


def ivf_build(vecs: np.ndarray, centroids: np.ndarray, codebooks=None):
    """Inverted lists over unit vectors [n, v].

    * cell of x = argmax_c <x, c> (unit keys and unit centroids: the same
      cell as the nearest centroid);
    * lists in cell order, members in ascending key index (offsets [nlist+1],
      ids [n]);
    * flat index: the member vectors in list order;
    * PQ index (codebooks [pq_m, 256, v / pq_m]): the residual r = x - c_cell
      is cut into pq_m sub-vectors and each is replaced by the index of its
      nearest codeword (L2, ties to the lowest index), as FAISS IVF-PQ
      encodes by residual.
    """
    x = np.asarray(vecs, F32)
    c = np.asarray(centroids, F32)
    nlist = c.shape[0]
    cell = assign_ip(x, c)
    ids = np.lexsort((np.arange(len(x)), cell)).astype(np.int32)
    cnt = np.bincount(cell, minlength=nlist)
    offsets = np.concatenate([[0], np.cumsum(cnt)]).astype(np.int64)
    out = {"offsets": offsets, "ids": ids, "cell": cell}
    if codebooks is None:
        out["vectors"] = x[ids]
        return out
    cb = np.asarray(codebooks, F32)
    pq_m, ksub, dsub = cb.shape
    r = (x - c[cell]).astype(F32)
    codes = np.zeros((len(x), pq_m), dtype=np.uint8)
    for m in range(pq_m):
        codes[:, m] = assign_l2(r[:, m * dsub:(m + 1) * dsub], cb[m])
    out["codes"] = codes[ids]
    return out


def ivf_search(index: dict, centroids: np.ndarray, queries: np.ndarray, nprobe: int, k: int,
               codebooks=None):
    """Top-k of the approximate scores over the nprobe best cells.

    * coarse score s_c = <q, c> (fp32); probe the nprobe largest, ties to the
      lower cell;
    * flat: score = <q, x>;
    * PQ: score = s_c + sum_m LUT[m][code_m] with LUT[m][b] = <q_m, B_m[b]>
      (inner product decomposes over the residual, as in FAISS IVF-PQ with
      the inner-product metric), m ascending;
    * top-k by (score desc, key index asc); fewer than k candidates leave
      score -inf and index -1 in the remaining slots.
    Returns (scores [q, k] f32, idx [q, k] int32, probes [q, nprobe] int32).
    """
    qv = np.asarray(queries, F32)
    c = np.asarray(centroids, F32)
    off, ids = index["offsets"], index["ids"]
    nq = qv.shape[0]
    coarse = dot_seq(qv[:, None, :], c[None, :, :])  # [q, nlist]
    out_s = np.full((nq, k), -np.inf, dtype=F32)
    out_i = np.full((nq, k), -1, dtype=np.int32)
    probes = np.zeros((nq, nprobe), dtype=np.int32)
    if codebooks is not None:
        cb = np.asarray(codebooks, F32)
        pq_m, ksub, dsub = cb.shape
    for qi in range(nq):
        order = np.lexsort((np.arange(c.shape[0]), -coarse[qi].astype(np.float64)))
        probes[qi] = order[:nprobe]
        cand_s, cand_i = [], []
        if codebooks is not None:
            lut = np.stack([dot_seq(qv[qi, m * dsub:(m + 1) * dsub][None, :], cb[m])
                            for m in range(pq_m)])  # [pq_m, 256]
        for cell in probes[qi]:
            lo, hi = off[cell], off[cell + 1]
            if hi == lo:
                continue
            if codebooks is None:
                s = dot_seq(qv[qi][None, :], index["vectors"][lo:hi])
            else:
                codes = index["codes"][lo:hi]
                s = np.full(hi - lo, coarse[qi, cell], dtype=F32)
                for m in range(pq_m):
                    s = (s + lut[m][codes[:, m]]).astype(F32)
            cand_s.append(s)
            cand_i.append(ids[lo:hi])
        if not cand_s:
            continue
        s = np.concatenate(cand_s)
        i = np.concatenate(cand_i)
        o = np.lexsort((i, -s.astype(np.float64)))[:k]
        out_s[qi, :len(o)] = s[o]
        out_i[qi, :len(o)] = i[o]
    return out_s, out_i, probes


def rescore_topk(keys_bits: np.ndarray, queries_bits: np.ndarray, cand: np.ndarray, k: int):
    """Exact similarity of each query's candidates, then its top k (Sec.
    3.2.2 Eq. 8: the approximate search returns N' candidates D_ret, the
    composite score ranks them by sim(h, k_i) between the full hidden state
    and each candidate's key, and Top-N keeps N of them).

    keys_bits [n, d] and queries_bits [q, d] bf16 bit patterns, cand [q, N']
    int key indices with -1 for an empty slot.  sim is the fp64 inner
    product of the stored bf16 values (``scores``).  The top k are ordered
    by (score desc, key index asc); slots beyond the valid candidates hold
    -inf / -1.  Returns (scores [q, k] f64, idx [q, k] int32).
    """
    cand = np.asarray(cand)
    nq = cand.shape[0]
    out_s = np.full((nq, k), -np.inf)
    out_i = np.full((nq, k), -1, dtype=np.int32)
    for qi in range(nq):
        c = cand[qi][cand[qi] >= 0].astype(np.int64)
        if c.size == 0:
            continue
        s = scores(np.asarray(keys_bits)[c], np.asarray(queries_bits)[qi:qi + 1])[0]
        order = np.lexsort((c, -s))[:k]
        out_s[qi, :order.size] = s[order]
        out_i[qi, :order.size] = c[order]
    return out_s, out_i


def recall_at_k(approx_idx: np.ndarray, exact_idx: np.ndarray) -> float:
    """Mean fraction of the exact top-k found in the approximate top-k."""
    hits = [len(set(a.tolist()) & set(e.tolist())) / len(e)
            for a, e in zip(approx_idx, exact_idx)]
    return float(np.mean(hits))
