"""Pins of the dynamic-context-buffer oracle (Alg. 1 R.Update, Alg. 2
DynSearch with the delta boost and the hybrid rerank): brute force over the
append history, invariances, special cases that reduce to the static path,
and a hand-worked hybrid list.  No GPU is needed."""
import numpy as np
import torch

import synth
from oracle import ctx_oracle as X
from oracle import sense_oracle as O


def _bits(t):
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def _history(T, d, vocab, seed):
    h = _bits(synth.gaussian_rows_f32(T, d, seed=seed).to(torch.bfloat16))
    tok = np.random.default_rng(seed).integers(0, vocab, T)
    return h, tok


def test_entries_bruteforce_ring():
    h, tok = _history(50, 32, 9, 1)
    for cap, m in ((64, 4), (20, 4), (8, 1), (5, 6)):
        for T in (0, 3, 6, 10, 50):
            pos, keys, spans = X.ctx_entries(h[:T], tok[:T], cap, m)
            want = [p for p in range(T) if p >= T - cap and p + m <= T]
            assert pos.tolist() == want
            for p, sp in zip(pos, spans):
                assert sp.tolist() == tok[p:p + m].tolist()
            if len(pos):
                np.testing.assert_array_equal(
                    keys, O.normalize_keys_bf16(O.bf16_bits_to_f64(h[pos]).astype(np.float32)))


def test_search_is_exact_topk_and_delta_shifts():
    h, tok = _history(300, 64, 50, 2)
    q = _bits(synth.gaussian_rows_f32(3, 64, seed=9).to(torch.bfloat16))
    s0, p0, sp0 = X.ctx_search(h, tok, 256, 5, q, 10, 0.0)
    s1, p1, sp1 = X.ctx_search(h, tok, 256, 5, q, 10, 0.75)
    np.testing.assert_array_equal(p0, p1)
    np.testing.assert_array_equal(sp0, sp1)
    np.testing.assert_allclose(s1, s0 + 0.75, rtol=0, atol=1e-15)
    pos, keys, spans = X.ctx_entries(h, tok, 256, 5)
    kf = O.bf16_bits_to_f64(keys)
    qf = O.bf16_bits_to_f64(q)
    for qi in range(3):
        dots = [(float(np.dot(qf[qi], kf[e])), -int(pos[e])) for e in range(len(pos))]
        best = sorted(range(len(pos)), key=lambda e: dots[e], reverse=True)[:10]
        assert p0[qi].tolist() == [int(pos[e]) for e in best]


def test_search_ties_go_to_older_position_and_short_buffer():
    h, tok = _history(12, 16, 7, 3)
    h[9] = h[2]  # equal keys at positions 2 and 9
    q = h[2:3].copy()
    s, p, sp = X.ctx_search(h, tok, 64, 3, q, 20, 0.0)
    assert p[0, 0] == 2 and p[0, 1] == 9
    n_entries = 12 - 3 + 1
    assert (p[0, n_entries:] == -1).all() and np.isneginf(s[0, n_entries:]).all()
    assert (sp[0, n_entries:] == -1).all()
    s, p, sp = X.ctx_search(h[:2], tok[:2], 64, 3, q, 4, 0.0)  # nothing searchable yet
    assert (p == -1).all()


def test_hybrid_reduces_to_static_and_orders_union():
    rng = np.random.default_rng(4)
    ks, kd, m = 6, 4, 3
    ss = np.sort(rng.uniform(0, 1, (2, ks)))[:, ::-1].copy()
    sp_s = rng.integers(0, 5, (2, ks, m)).astype(np.int32)
    sp_d = rng.integers(0, 5, (2, kd, m)).astype(np.int32)
    empty = np.full((2, kd), -np.inf)
    anchor = np.array([1, 3])
    # no dynamic results: the static path (gather with rerank on rank order)
    got = X.hybrid_drafts(ss, sp_s, empty, sp_d, anchor, 5, True)
    table = sp_s.reshape(2 * ks, m)
    idx = np.arange(2 * ks).reshape(2, ks)
    want = O.gather_drafts(table, idx, anchor, 5, True)
    np.testing.assert_array_equal(got, want)
    # a large boost puts every dynamic result ahead of the static ones
    ds_ = np.sort(rng.uniform(0, 1, (2, kd)))[:, ::-1] + 10.0
    got = X.hybrid_drafts(ss, sp_s, ds_, sp_d, None, ks + kd)
    np.testing.assert_array_equal(got[:, :kd], sp_d)
    np.testing.assert_array_equal(got[:, kd:], sp_s)


def test_hybrid_hand_worked():
    # static scores 0.9, 0.5 with first tokens 7, 4; dynamic (boosted) 0.7,
    # 0.5 with first tokens 4, 9; anchor 4.  Union by score with ties static
    # first: S0(.9,7) D0(.7,4) S1(.5,4) D1(.5,9); anchor-first: D0, S1, S0, D1;
    # keep 3 and force the anchor into the first token of rows 0 and 2.
    ss = np.array([[0.9, 0.5]])
    sp_s = np.array([[[7, 1], [4, 2]]])
    ds_ = np.array([[0.7, 0.5]])
    sp_d = np.array([[[4, 3], [9, 5]]])
    got = X.hybrid_drafts(ss, sp_s, ds_, sp_d, np.array([4]), 3, True)
    assert got[0].tolist() == [[4, 3], [4, 2], [4, 1]]
