"""Plain CPU oracle for the SENSE drafting hot path (test infrastructure only).

This module is the slow, obviously-correct reference that the CUDA library is
checked against.  It is TEST INFRASTRUCTURE: only the test suite, the smoke
check in ``__graft_entry__`` and the ``cpu_baseline`` / ``--impl reference``
legs of ``bench.py`` may import it.  The product path never calls it, and it
shares no code with the CUDA library (no helpers, tables or constants).

Every function below restates one step of SENSE ("Semantic Embedding
Navigation with Soft-gated Evaluation", arxiv 2606.00021) in numpy, in fp64
for floating point, following the step order and notation of the paper:

  normalize_keys_bf16  §3.2.1 Eq. 6 + App. E "Datastore Construction"
                        (L2-normalised keys), stored as bf16
  scores               §3.2.2 Eq. 8 sim(.,.) / App. C.2 Alg. 2 (inner product
                        of unit-norm vectors)
  topk                 §3.2.2 Eq. 7 (top-N' by similarity), exact search
  gather_drafts        §3.2.2 D_ret = {(k_i, s_i)}, Eq. 8 composite rerank,
                        Alg. 2 forced anchor
  loose_trie           §3.2.3 Eq. 9 (sorted-LCP trie), node-capped
  loose_trie_alg3      App. C.3 Alg. 3 restated step by step (uncapped)
  mask_from_bits,      App. C.6 Eq. 20 (additive tree attention mask over a
  tree_mask_full        static KV cache) from Alg. 3's mask M
  tree_attention       the masked attention of the verify forward (Alg. 1)
                        under that mask
  soft_gate            §3.3 Eqs. 11-19 (with App. C.4's normalised entropy
                        and look-ahead window)

Readings where the paper is silent or ambiguous are stated at each function.

Pins: every function is pinned by tests under ``tests/`` (brute force on tiny
inputs, closed forms, invariants, library special cases).  No function here
is "parity unpinned".
"""
from __future__ import annotations

import math

import numpy as np

# ----------------------------------------------------------------------------
# bf16 encoding (the storage type of the datastore keys)
# ----------------------------------------------------------------------------


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Decode bf16 bit patterns (uint16) to float64, exactly.

    A bf16 value is the upper half of an IEEE-754 binary32 word, so widening
    the 16 bits to the top of a 32-bit word gives the same number as float32,
    which float64 represents exactly.
    """
    b = np.ascontiguousarray(bits).view(np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def f64_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float64 values to the nearest bf16 (ties to even), return bits.

    bf16 has an 8-bit significand (7 stored bits) and the binary32 exponent
    range, so for |x| >= 2^-126 its spacing near x is 2^(e-7) with
    e = floor(log2 |x|); below that (subnormal range) the spacing is 2^-133.
    The value is divided by that spacing, rounded half-to-even (np.rint), and
    scaled back; the result is exactly representable in binary32.
    Overflow saturates to +-inf, as round-to-nearest does.
    """
    x = np.asarray(x, dtype=np.float64)
    out = np.zeros(x.shape, dtype=np.float64)
    a = np.abs(x)
    nz = a > 0
    e = np.floor(np.log2(np.where(nz, a, 1.0)))
    # log2 of a value just below a power of two may round up: correct e.
    e = np.where(np.ldexp(1.0, e.astype(np.int64)) > a, e - 1, e)
    e = np.maximum(e, -126.0)
    ulp = np.ldexp(1.0, (e - 7).astype(np.int64))
    r = np.rint(x / ulp) * ulp
    out = np.where(nz, r, x)  # keeps signed zero
    max_bf16 = (2.0 - 2.0 ** -7) * 2.0 ** 127
    out = np.where(np.abs(out) > max_bf16, np.copysign(np.inf, out), out)
    f32 = out.astype(np.float32)
    return (f32.view(np.uint32) >> 16).astype(np.uint16)


# ----------------------------------------------------------------------------
# a1: datastore keys (§3.2.1 Eq. 6; App. E "Datastore Construction")
# ----------------------------------------------------------------------------


def normalize_keys_bf16(keys_f32: np.ndarray) -> np.ndarray:
    """Unit-L2-normalise each key row and store it as bf16 (bits, uint16).

    §3.2.1 Eq. 6 stores keys Z(h); App. E states the projected embeddings are
    L2-normalised before indexing.  Each row x becomes x / ||x||_2 computed in
    fp64, then rounded once to bf16 (round to nearest, ties to even).
    Reading: a zero row has no direction; it is stored as zeros.
    """
    x = np.asarray(keys_f32, dtype=np.float64)
    norm = np.sqrt(np.sum(x * x, axis=1, keepdims=True))
    y = np.where(norm > 0, x / np.where(norm > 0, norm, 1.0), 0.0)
    return f64_to_bf16_bits(y)


# ----------------------------------------------------------------------------
# a2: scoring (§3.2.2 Eq. 8 sim(.,.); Alg. 2 L2Norm then search)
# ----------------------------------------------------------------------------


def scores(keys_bits: np.ndarray, queries_bits: np.ndarray,
           chunk: int = 16384) -> np.ndarray:
    """s[q, i] = <query_q, key_i> in fp64 over the stored bf16 values.

    The similarity of §3.2.2 Eq. 8 between unit-norm vectors (Alg. 2 applies
    L2Norm to the query; App. E normalises the keys) is their inner product.
    The stored bf16 keys are used as stored (not renormalised).  Keys are
    widened to fp64 in row chunks so the working set stays bounded; each
    chunk is one matrix product.
    """
    qf = bf16_bits_to_f64(queries_bits)
    n = keys_bits.shape[0]
    out = np.empty((qf.shape[0], n), dtype=np.float64)
    for lo in range(0, n, chunk):
        hi = min(n, lo + chunk)
        kf = bf16_bits_to_f64(keys_bits[lo:hi])
        out[:, lo:hi] = qf @ kf.T
    return out


# ----------------------------------------------------------------------------
# a3: top-k (§3.2.2 Eq. 7, exact search)
# ----------------------------------------------------------------------------


def topk(score_rows: np.ndarray, k: int):
    """The k highest scores of each row, by (score desc, index asc).

    §3.2.2 Eq. 7 retrieves the top-N' keys by similarity.  Reading: the
    search is exact (not approximate); ties are broken by the lower key
    index, which makes the order total.
    Returns (values [Q, k] float64, indices [Q, k] int64).
    """
    s = np.atleast_2d(np.asarray(score_rows, dtype=np.float64))
    qn, n = s.shape
    if not (1 <= k <= n):
        raise ValueError("need 1 <= k <= n")
    vals = np.empty((qn, k), dtype=np.float64)
    idxs = np.empty((qn, k), dtype=np.int64)
    for q in range(qn):
        row = s[q]
        # Every index whose score is >= the k-th largest value is a candidate;
        # ties at that value are all kept, then the total order decides.
        kth = np.partition(row, n - k)[n - k]
        cand = np.nonzero(row >= kth)[0]
        order = np.lexsort((cand, -row[cand]))  # primary: -score, then index
        pick = cand[order[:k]]
        vals[q] = row[pick]
        idxs[q] = pick
    return vals, idxs


# ----------------------------------------------------------------------------
# a4: gather of continuation spans (+ composite rerank and forced anchor)
# ----------------------------------------------------------------------------


def gather_drafts(spans: np.ndarray, idx: np.ndarray, anchor=None,
                  n_keep: int | None = None, force_anchor: bool = False):
    """Candidate spans D[q, r, :] = spans[idx[q, r], :].

    §3.2.2 defines D_ret = {(k_i, s_i)}: each retrieved key brings its stored
    continuation span.  An index outside [0, N) yields a row of -1.

    With an anchor token x~ per query, Eq. 8 rescores each candidate as
    S = alpha * I(s[0] == x~) + beta * sim with alpha >> beta and keeps the
    Top-N.  Reading: alpha >> beta makes this the lexicographic order
    (anchor match first, then retrieval rank, which is the similarity
    order), i.e. a stable partition of the retrieved list; the first n_keep
    rows are kept.  With ``force_anchor`` the first token of the first kept
    row and of the last kept row are set to x~ (Alg. 2 forces the anchor
    into the first token of the first and of the last candidate).
    """
    spans = np.asarray(spans)
    idx = np.atleast_2d(np.asarray(idx, dtype=np.int64))
    qn, k = idx.shape
    m = spans.shape[1]
    n = spans.shape[0]
    raw = np.full((qn, k, m), -1, dtype=np.int32)
    for q in range(qn):
        for r in range(k):
            i = idx[q, r]
            if 0 <= i < n:
                raw[q, r] = spans[i]
    if anchor is None:
        return raw
    anchor = np.asarray(anchor, dtype=np.int64).reshape(qn)
    keep = k if n_keep is None else int(n_keep)
    out = np.empty((qn, keep, m), dtype=np.int32)
    for q in range(qn):
        valid = (idx[q] >= 0) & (idx[q] < n)
        match = valid & (raw[q, :, 0] == anchor[q])
        order = [r for r in range(k) if match[r]] + \
                [r for r in range(k) if not match[r]]
        out[q] = raw[q, order[:keep]]
        if force_anchor and keep > 0:
            out[q, 0, 0] = anchor[q]
            out[q, keep - 1, 0] = anchor[q]
    return out


# ----------------------------------------------------------------------------
# a5: loose trie (§3.2.3 Eq. 9; App. C.3 Alg. 3)
# ----------------------------------------------------------------------------


def loose_trie(spans_qkm: np.ndarray, node_cap: int = 0, mask_bits=False):
    """Deduplicated prefix tree of the candidate spans of each query.

    §3.2.3 Eq. 9 sorts the candidates lexicographically and emits, for each
    sorted row, the tokens after its longest common prefix with the previous
    row; App. C.3 Alg. 3 does the same with masks.  The emitted sequence is
    the set of distinct non-empty prefixes of the candidates, listed in
    lexicographic preorder.  This function computes that set directly:

    * node = distinct non-empty prefix s_r[0..j] of some candidate row r;
    * node ids follow lexicographic order of the token paths (a prefix sorts
      before its extensions), which is the order of T_flat in Eq. 9;
    * parent = the prefix one token shorter (-1 for depth 0: a child of the
      current position); depth is 0-based;
    * gamma[r, j] = id of s_r[0..j] (the mapping Gamma of Alg. 3), indexed
      by input rank r (Alg. 3 returns it in sorted order; here it is
      permuted back to the candidates' order);
    * ancestor-or-self mask (Alg. 3's M) as bits: bit b of row n is set iff
      node b lies on the root path of node n.

    Reading (the paper sets no cap): with ``node_cap`` C > 0 each node gets
    the key (first_rank, depth), first_rank being the smallest input rank r
    having that prefix; the C smallest keys are kept.  A parent's key is
    strictly smaller than its child's, so the kept set is prefix-closed;
    positions whose node is dropped get gamma = -1.  Output arrays are sized
    C (or k*M when uncapped) and padded with -1.

    Tokens must be >= 0 (negative ids are reserved as padding).
    Returns a dict of numpy arrays with a leading query axis.
    """
    s = np.asarray(spans_qkm, dtype=np.int64)
    if s.ndim == 2:
        s = s[None]
    qn, k, m = s.shape
    if np.any(s < 0):
        raise ValueError("token ids must be >= 0")
    cap = node_cap if node_cap > 0 else k * m
    words = (cap + 31) // 32
    res = {
        "num_nodes": np.zeros(qn, dtype=np.int32),
        "tokens": np.full((qn, cap), -1, dtype=np.int32),
        "parent": np.full((qn, cap), -1, dtype=np.int32),
        "depth": np.full((qn, cap), -1, dtype=np.int32),
        "gamma": np.full((qn, k, m), -1, dtype=np.int32),
    }
    if mask_bits:
        res["mask_bits"] = np.zeros((qn, cap, words), dtype=np.uint32)
    for q in range(qn):
        first_rank = {}
        for r in range(k):
            for j in range(m):
                p = tuple(int(t) for t in s[q, r, :j + 1])
                if p not in first_rank:
                    first_rank[p] = r
        by_key = sorted(first_rank, key=lambda p: (first_rank[p], len(p)))
        kept = set(by_key[:cap])
        order = sorted(kept)  # tuple order: lexicographic, prefix first
        nid = {p: i for i, p in enumerate(order)}
        res["num_nodes"][q] = len(order)
        for p, i in nid.items():
            res["tokens"][q, i] = p[-1]
            res["depth"][q, i] = len(p) - 1
            res["parent"][q, i] = nid[p[:-1]] if len(p) > 1 else -1
        for r in range(k):
            for j in range(m):
                p = tuple(int(t) for t in s[q, r, :j + 1])
                res["gamma"][q, r, j] = nid.get(p, -1)
        if mask_bits:
            for p, i in nid.items():
                for j in range(1, len(p) + 1):
                    b = nid[p[:j]]
                    res["mask_bits"][q, i, b // 32] |= np.uint32(1 << (b % 32))
    return res


def loose_trie_alg3(d_sorted_or_not: np.ndarray):
    """App. C.3 Alg. 3's vectorised trie, in its order (one query, no node cap).

    The rows are put in lexicographic order first (Alg. 2 sorts before it
    builds).  A cell (i, j) repeats an earlier node exactly when row i agrees
    with row i-1 on every column up to and including j; the other cells are
    new nodes, numbered in row-major reading order, which is preorder.  A
    repeated cell takes the number of the latest new node above it in its
    column (a running maximum down the column), and the ancestor mask marks,
    for every row, each of its nodes against every earlier node on the same
    row.  Returns (tokens of the new cells, Gamma in sorted-row order, the
    mask, the sort permutation pi).
    """
    d = np.asarray(d_sorted_or_not, dtype=np.int64)
    n, m = d.shape
    # LexSort: np.lexsort uses its LAST key as primary, so pass columns
    # reversed; equal rows keep their input order (stable).
    pi = np.lexsort(tuple(d[:, j] for j in range(m - 1, -1, -1)))
    ds = d[pi]
    match = np.zeros((n, m), dtype=np.int64)
    match[1:] = (ds[1:] == ds[:-1]).astype(np.int64)
    is_prefix = np.cumprod(match, axis=1)
    unique = is_prefix == 0
    t_flat = ds[unique]
    big_l = t_flat.shape[0]
    idx = np.cumsum(unique.reshape(-1)) - 1
    gam = idx.reshape(n, m)
    tmp = np.where(unique, gam, -1)
    gam = np.maximum.accumulate(tmp, axis=0)
    mask = np.zeros((big_l, big_l), dtype=np.int64)
    ii, jj = np.tril_indices(m)
    for i in range(n):
        mask[gam[i, ii], gam[i, jj]] = 1
    return t_flat, gam, mask, pi


# ----------------------------------------------------------------------------
# tree attention mask over a static KV cache (App. C.6 Eq. 20)
# ----------------------------------------------------------------------------


def mask_from_bits(bits_rows: np.ndarray, num_nodes: int) -> np.ndarray:
    """Alg. 3's 0/1 draft mask M (L x L) from ancestor bit rows.

    ``bits_rows[n, w]`` holds bits 32w..32w+31 of row n (the layout of
    ``loose_trie(..., mask_bits=True)``): M[n, b] = bit b of row n.
    """
    b = np.asarray(bits_rows)
    big_l = int(num_nodes)
    out = np.zeros((big_l, big_l), dtype=np.int64)
    for n in range(big_l):
        for c in range(big_l):
            out[n, c] = (int(b[n, c // 32]) >> (c % 32)) & 1
    return out


def tree_mask_full(M: np.ndarray, m: int, cache_len: int, rows=None) -> np.ndarray:
    """Additive attention mask M_full of App. C.6 Eq. 20, fp64.

    The L draft tokens sit at cache positions m..m+L-1 behind m committed
    tokens, in a static cache of cache_len positions.  Row i (draft token i)
    gets 0 at column j when j < m (every committed token is visible) or when
    m <= j < m+L and M[i, j-m] = 1 (an ancestor-or-self tree token), and
    -inf everywhere else.

    Reading: ``rows`` >= L pads the output for a fixed node capacity; a
    padding row has no tree entries, so the same rule gives it 0 on the
    committed columns and -inf elsewhere.  m + L must fit in the cache.
    """
    big_m = np.asarray(M)
    big_l = big_m.shape[0]
    rows = big_l if rows is None else int(rows)
    if m < 0 or m + big_l > cache_len or rows < big_l:
        raise ValueError("need 0 <= m, m + L <= cache_len and rows >= L")
    out = np.full((rows, cache_len), -np.inf)
    out[:, :m] = 0.0
    for i in range(big_l):
        for c in range(big_l):
            if big_m[i, c] == 1:
                out[i, m + c] = 0.0
    return out


def tree_attention(q_bits: np.ndarray, k_bits: np.ndarray, v_bits: np.ndarray, m: int,
                   M: np.ndarray, scale: float) -> np.ndarray:
    """Tree-masked attention of the L draft tokens over a static KV cache, fp64.

    The verify forward of Alg. 1 (Forward(T, M_full, K)) scores every draft
    token against the cache under the additive mask M_full of Eq. 20:
    O[h] = softmax(scale * Q[h] K[h]^T + M_full) V[h] over the first m + L
    cache positions.  q_bits [H, L, D], k_bits / v_bits [H, >= m + L, D]
    (bf16 bits); M [L, L] is Alg. 3's 0/1 mask.  Returns [H, L, D].
    """
    qf = bf16_bits_to_f64(np.asarray(q_bits))
    kf = bf16_bits_to_f64(np.asarray(k_bits))
    vf = bf16_bits_to_f64(np.asarray(v_bits))
    big_l = qf.shape[1]
    n = m + big_l
    full = tree_mask_full(M, m, n)
    out = np.empty_like(qf)
    for h in range(qf.shape[0]):
        s = scale * (qf[h] @ kf[h, :n].T) + full
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p /= p.sum(axis=1, keepdims=True)
        out[h] = p @ vf[h, :n]
    return out


# ----------------------------------------------------------------------------
# a6: soft-gated evaluation (§3.3 Eqs. 11-19; App. C.4 Alg. 4)
# ----------------------------------------------------------------------------


def _softmax_entropy(rows: np.ndarray) -> np.ndarray:
    """Shannon entropy (nats) of softmax(rows) along the last axis, fp64:
    -sum_v p_v log p_v over the softmax probabilities p (0 log 0 = 0), the
    entropy of Eq. 14 taken of the logits' distribution as App. C.4 does.
    """
    x = np.asarray(rows, dtype=np.float64)
    z = x - x.max(axis=-1, keepdims=True)
    e = np.exp(z)
    p = e / e.sum(axis=-1, keepdims=True)
    with np.errstate(divide="ignore", invalid="ignore"):
        plogp = np.where(p > 0, p * np.log(np.where(p > 0, p, 1.0)), 0.0)
    return -plogp.sum(axis=-1)


def _in_topk(rows: np.ndarray, tok: np.ndarray, kappa: int) -> np.ndarray:
    """I(tok in TopK(row, kappa)) with the total order (value desc, index asc).

    Eq. 15's top-k set does not say how ties at its boundary are broken.
    Reading: the lower vocabulary index wins, so the token is in the
    top-kappa iff fewer than kappa entries precede it in that order.
    """
    x = np.asarray(rows, dtype=np.float32)
    v = x.shape[-1]
    t = np.clip(tok, 0, v - 1)
    xt = np.take_along_axis(x, t[..., None], axis=-1)
    ar = np.arange(v)
    ahead = (x > xt) | ((x == xt) & (ar < t[..., None]))
    return (ahead.sum(axis=-1) < kappa) & (tok >= 0) & (tok < v)


def soft_gate(tokens, parent, num_nodes, gamma, root_logits, node_logits,
              root_hidden, node_hidden, *, gamma_thr=0.05, kappa=3, window=6,
              tau=0, unnormalized_entropy=False, return_masks=False,
              ent_band=0.0):
    """Soft-gated evaluation of every candidate path of every query (§3.3).

    Inputs per query q (leading axis): the tree (tokens, parent, num_nodes,
    gamma [k, M]) and the target outputs on it: root_logits [V] = p (the
    state before the draft), node_logits [cap, V] = P' (one row per tree
    node), root_hidden [d] = h, node_hidden [cap, d] = H'.

    Candidate i is the path of nodes gamma[i, 0], gamma[i, 1], ...; its draft
    token at position j is D[i, j] = tokens[gamma[i, j]].  The target's
    prediction for position j comes from the state just before it (Eq. 11,
    the alignment that prepends p and h): the root row p for j = 0 and the
    row of node gamma[i, j-1] otherwise.  (The printed shape "M x (N+1)" is
    read as N candidates, each with its root row plus M positions.)

    For each position (i, j), with r its predicting row:
      * Eq. 12-13: em = 1 when D[i, j] is the greedy token of r (the lowest
        index among equal maxima);
      * Eq. 14: ent = 1 when the entropy of softmax(r), in nats and divided
        by log|V|, exceeds gamma_thr (the normalisation is App. C.4's;
        ``unnormalized_entropy`` compares the raw entropy as Eq. 14 prints);
      * Eq. 15: topk = 1 when fewer than kappa vocabulary entries come before
        D[i, j] in the order (value desc, index asc) of r;
      * Eq. 16: con = 1 when the positions j+1 .. j+W of the same candidate
        hold at most tau mismatches (1 - em), positions past the span
        counting as mismatches (the window looks strictly ahead: App. C.4
        pads with ones on the right and drops the first output);
      * Eq. 17: G = em or (ent and (topk or con)).
    Eq. 18: n_i is the number of leading ones of G[i, :], the accepted
    length; L_i = n_i - 1 (App. C.4 and Alg. 1 index the accepted tokens
    D[i, 0 .. L_i]); i* is the lowest candidate rank with the largest L_i.
    Positions whose node was dropped by the tree's node cap (gamma = -1)
    have em = ent = topk = G = 0 and count as mismatches inside a window.

    Next state (Eq. 19; Alg. 1): accepted tokens a = D[i*, 0 .. L*]; the next
    node is gamma[i*, L*] (-1, the root, when L* = -1); h_next is that
    node's hidden state (h when -1) and p_next its logits row, whose greedy
    token is the next anchor.

    ``ent_band`` > 0 also reports, per query, whether any evaluated
    position had a normalised entropy within ``ent_band`` of the threshold
    (such decisions depend on rounding and are excluded from parity).
    """
    tokens = np.asarray(tokens)
    parent = np.asarray(parent)
    gamma = np.asarray(gamma)
    root_logits = np.asarray(root_logits, dtype=np.float32)
    node_logits = np.asarray(node_logits, dtype=np.float32)
    root_hidden = np.asarray(root_hidden)
    node_hidden = np.asarray(node_hidden)
    qn, k, m = gamma.shape
    v = root_logits.shape[-1]
    w = int(window)
    out = {
        "i_star": np.zeros(qn, dtype=np.int32),
        "L_star": np.zeros(qn, dtype=np.int32),
        "n_accept": np.zeros(qn, dtype=np.int32),
        "accepted": np.full((qn, m), -1, dtype=np.int32),
        "next_node": np.zeros(qn, dtype=np.int32),
        "next_anchor": np.zeros(qn, dtype=np.int32),
        "h_next": np.zeros((qn,) + root_hidden.shape[1:], dtype=root_hidden.dtype),
        "G": np.zeros((qn, k, m), dtype=np.uint8),
        "ambiguous": np.zeros(qn, dtype=bool),
    }
    if return_masks:
        for key in ("B_em", "B_ent", "B_topk", "B_con"):
            out[key] = np.zeros((qn, k, m), dtype=np.uint8)
    for q in range(qn):
        g = gamma[q].astype(np.int64)
        kept = g >= 0
        em = np.zeros((k, m), dtype=bool)
        ent = np.zeros((k, m), dtype=bool)
        top = np.zeros((k, m), dtype=bool)
        amb = False
        for i in range(k):
            for j in range(m):
                if not kept[i, j]:
                    continue
                tok = int(tokens[q, g[i, j]])
                row = root_logits[q] if j == 0 else node_logits[q, g[i, j - 1]]
                em[i, j] = tok == int(np.argmax(row))  # first maximum
                h = _softmax_entropy(row)
                score = h if unnormalized_entropy else h / math.log(v)
                ent[i, j] = score > gamma_thr
                if ent_band > 0 and abs(score - gamma_thr) < ent_band:
                    amb = True
                top[i, j] = bool(_in_topk(row, np.array(tok), kappa))
        # mismatch indicator per position; dropped positions and the
        # positions past the span (j >= M) are mismatches
        miss = ~(em & kept)
        con = np.zeros((k, m), dtype=bool)
        for i in range(k):
            for j in range(m):
                ahead = [bool(miss[i, u]) if u < m else True for u in range(j + 1, j + w + 1)]
                con[i, j] = kept[i, j] and sum(ahead) <= tau
        gmask = (em | (ent & (top | con))) & kept
        n_acc = np.zeros(k, dtype=np.int64)
        for i in range(k):
            while n_acc[i] < m and gmask[i, n_acc[i]]:
                n_acc[i] += 1
        li = n_acc - 1
        istar = int(np.argmax(li))  # the first (lowest rank) maximum
        lstar = int(li[istar])
        out["i_star"][q] = istar
        out["L_star"][q] = lstar
        out["n_accept"][q] = lstar + 1
        for j in range(lstar + 1):
            out["accepted"][q, j] = tokens[q, g[istar, j]]
        nxt = int(g[istar, lstar]) if lstar >= 0 else -1
        out["next_node"][q] = nxt
        prow = root_logits[q] if nxt < 0 else node_logits[q, nxt]
        out["next_anchor"][q] = int(np.argmax(prow))
        out["h_next"][q] = root_hidden[q] if nxt < 0 else node_hidden[q, nxt]
        out["G"][q] = gmask.astype(np.uint8)
        out["ambiguous"][q] = amb
        if return_masks:
            out["B_em"][q] = em
            out["B_ent"][q] = ent & kept
            out["B_topk"][q] = top & kept
            out["B_con"][q] = con
    return out
