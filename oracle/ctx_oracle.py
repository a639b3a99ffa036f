"""Plain CPU oracle of the dynamic context buffer (test infrastructure only).

Only the test suite, the smoke check and the CPU legs of the benchmark import
this module; the product library never uses it and shares no code with it.

SENSE retrieves from a hybrid store C_db = C_s u C_d (Sec. 3.2.1 Eq. 6): the
static corpus C_s and a dynamic buffer C_d filled from the generation itself.
Alg. 1 fills it with R.Update(h, y) after prefill and R.Update(H_align[i*,
0:L*+1], a) after every accepted step: pairs of a hidden state and the token
it predicted.  Alg. 2 searches it with DynSearch(h, C_d, x~), adds a score
boost delta to its results (s = [s_s; s_d + delta]) and reranks the union
with Eq. 8.  The paper does not define DynSearch or the buffer's size; this
module reads them as follows:

* an entry is a position p of the generated sequence: its key is the hidden
  state h_p that predicted token y_{p+1}, L2-normalised and stored as bf16
  (like the static keys, App. E), and its continuation span is
  y_{p+1} .. y_{p+M};
* a position becomes searchable once its M continuation tokens exist, and the
  buffer keeps the C most recent positions (a ring);
* DynSearch is the exact inner-product top-k over the searchable entries
  (ties to the older position), and its scores carry the boost delta;
* the hybrid candidate list orders the union by boosted score (ties keep the
  static results first, in rank order) and then applies the anchor rerank and
  forced anchor of Eq. 8 / Alg. 2 exactly as for static results.
"""
from __future__ import annotations

import numpy as np

from .sense_oracle import bf16_bits_to_f64, gather_drafts, normalize_keys_bf16, scores


def ctx_entries(hidden_bits: np.ndarray, tokens: np.ndarray, capacity: int, m: int):
    """Searchable entries after appending positions 0..T-1.

    hidden_bits [T, d] uint16 (bf16 hidden states h_p), tokens [T] int (the
    token y_{p+1} that h_p predicted, i.e. the sequence shifted by one).
    Returns (positions [E] int64, keys [E, d] uint16 bf16, spans [E, m]).
    """
    h = np.asarray(hidden_bits)
    tok = np.asarray(tokens, dtype=np.int64)
    total = h.shape[0]
    lo = max(0, total - capacity)
    hi = total - m + 1  # span of p = tok[p .. p+m-1] must exist: p + m - 1 <= total - 1
    pos = np.arange(lo, max(lo, hi), dtype=np.int64)
    keys = normalize_keys_bf16(bf16_bits_to_f64(h[pos]).astype(np.float32)) if len(pos) else \
        np.zeros((0, h.shape[1]), np.uint16)
    spans = np.stack([tok[p:p + m] for p in pos]) if len(pos) else np.zeros((0, m), np.int64)
    return pos, keys, spans.astype(np.int32)


def ctx_search(hidden_bits, tokens, capacity: int, m: int, query_bits, k: int, delta: float):
    """DynSearch: exact top-k of <q, key> + delta over the searchable entries,
    order (score desc, position asc).  Slots past the number of entries get
    score -inf, position -1 and a span of -1.
    Returns (scores [q, k] f64, positions [q, k] int64, spans [q, k, m] int32).
    """
    pos, keys, spans = ctx_entries(hidden_bits, tokens, capacity, m)
    qb = np.atleast_2d(np.asarray(query_bits))
    nq = qb.shape[0]
    out_s = np.full((nq, k), -np.inf)
    out_p = np.full((nq, k), -1, dtype=np.int64)
    out_sp = np.full((nq, k, m), -1, dtype=np.int32)
    if len(pos) == 0:
        return out_s, out_p, out_sp
    s = scores(keys, qb) + delta  # [q, E]
    for qi in range(nq):
        o = np.lexsort((pos, -s[qi]))[:k]
        out_s[qi, :len(o)] = s[qi, o]
        out_p[qi, :len(o)] = pos[o]
        out_sp[qi, :len(o)] = spans[o]
    return out_s, out_p, out_sp


def hybrid_drafts(static_scores, static_spans, dyn_scores, dyn_spans, anchor=None,
                  n_keep=None, force_anchor=False):
    """Candidate drafts from the union of static and dynamic results.

    static_scores [q, ks], static_spans [q, ks, m]; dyn_scores [q, kd]
    (already boosted by delta; -inf marks an empty slot), dyn_spans
    [q, kd, m].  The union is ordered by score (desc), ties keeping static
    before dynamic and rank order within each; empty dynamic slots are
    dropped (they sort last and are never kept ahead of a real candidate).
    Then Eq. 8's anchor-first rerank and Alg. 2's forced anchor apply as in
    ``gather_drafts``.  Returns int32 [q, n_keep, m].
    """
    ss = np.atleast_2d(np.asarray(static_scores, dtype=np.float64))
    ds_ = np.atleast_2d(np.asarray(dyn_scores, dtype=np.float64))
    sp_s = np.asarray(static_spans)
    sp_d = np.asarray(dyn_spans)
    nq, ks = ss.shape
    kd = ds_.shape[1]
    m = sp_s.shape[2]
    keep = ks + kd if n_keep is None else int(n_keep)
    out = np.empty((nq, keep, m), dtype=np.int32)
    for qi in range(nq):
        s = np.concatenate([ss[qi], ds_[qi]])
        table = np.concatenate([sp_s[qi], sp_d[qi]]).astype(np.int32)
        live = np.isfinite(s)
        order = np.lexsort((np.arange(ks + kd), -np.where(live, s, -np.inf)))
        order = [int(i) for i in order if live[i]]
        idx = np.full(ks + kd, -1, dtype=np.int64)
        idx[:len(order)] = order
        a = None if anchor is None else np.asarray(anchor).reshape(nq)[qi:qi + 1]
        rows = gather_drafts(table, idx[None, :], a, keep, force_anchor)
        out[qi] = rows[0, :keep]
    return out
