"""Pins of the approximate-retrieval oracle (PCA projection, k-means, IVF
flat / IVF-PQ) to facts fixed by the paper and by mathematics: fp64 error
bounds, brute force, special cases that reduce to exhaustive search, Lloyd's
monotone objective, and the hand-worked index in tests/golden/ivf_small.json.
No GPU is needed."""
import json
import os

import numpy as np
import pytest
import torch

import synth
from oracle import ivf_oracle as I
from oracle import sense_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
U = 2.0 ** -24  # fp32 unit roundoff


def _bits(t):
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def _unit(rng, n, d):
    x = rng.standard_normal((n, d))
    return (x / np.linalg.norm(x, axis=1, keepdims=True)).astype(np.float32)


# ---------------------------------------------------------------- reductions

def test_dot_and_l2_within_fp32_error_bound():
    rng = np.random.default_rng(1)
    a = rng.standard_normal((200, 64)).astype(np.float32)
    b = rng.standard_normal((200, 64)).astype(np.float32)
    ex = np.sum(a.astype(np.float64) * b, axis=1)
    bound = 64 * U * np.sum(np.abs(a.astype(np.float64) * b), axis=1) * 1.01
    assert np.all(np.abs(I.dot_seq(a, b) - ex) <= bound)
    ex2 = np.sum((a.astype(np.float64) - b) ** 2, axis=1)
    assert np.all(np.abs(I.l2_seq(a, b) - ex2) <= 66 * U * ex2 * 1.01)


def test_dot_exact_on_dyadic_values_and_order_matters():
    rng = np.random.default_rng(2)
    a = (rng.integers(-8, 9, (50, 32)) / 16).astype(np.float32)
    b = (rng.integers(-8, 9, (50, 32)) / 16).astype(np.float32)
    np.testing.assert_array_equal(I.dot_seq(a, b), (a.astype(np.float64) * b).sum(1))
    # the stated order is left to right: 1 + 2^-24 rounds back to 1 (ties to
    # even), while -1 + 2^-24 + 2^-24 + 1 keeps both small terms
    x = np.array([[1.0, 2 ** -24, 2 ** -24, -1.0]], np.float32)
    assert I.dot_seq(x, np.ones_like(x))[0] == 0.0
    assert I.dot_seq(x[:, ::-1].copy(), np.ones_like(x))[0] == 2.0 ** -23


# ---------------------------------------------------------------- projection

def test_project_exact_on_dyadic_inputs():
    """Small dyadic inputs: every product and sum is a short binary fraction,
    so the fp64 result must equal exact rational arithmetic."""
    from fractions import Fraction as F
    rng = np.random.default_rng(3)
    n, d, v = 4, 24, 5
    xv = rng.integers(-6, 7, (n, d)) / 8.0
    x = torch.tensor(xv, dtype=torch.float32).to(torch.bfloat16)
    xb = _bits(x)
    w = (rng.integers(-9, 10, (v, d)) / 16.0).astype(np.float32)
    mu = (rng.integers(-3, 4, d) / 4.0).astype(np.float32)
    y = I.project(xb, w, mu, normalize=False)
    for i in range(n):
        for o in range(v):
            ex = sum((F(float(xv[i, j])) - F(float(mu[j]))) * F(float(w[o, j])) for j in range(d))
            assert F(float(y[i, o])) == ex


def test_project_coordinate_basis_and_zero_row():
    x = synth.gaussian_rows_f32(6, 64, seed=4).to(torch.bfloat16)
    xb = _bits(x)
    sel = [5, 0, 63, 17]
    w = np.eye(64, dtype=np.float32)[sel]
    y = I.project(xb, w, normalize=False)
    np.testing.assert_array_equal(y, O.bf16_bits_to_f64(xb)[:, sel])
    # a signed permutation of coordinates only permutes and flips them
    w2 = -np.eye(64, dtype=np.float32)[sel[::-1]]
    np.testing.assert_array_equal(I.project(xb, w2, normalize=False), -y[:, ::-1])
    # centring on the row itself gives a zero row, left at zero by the norm
    mu = O.bf16_bits_to_f64(xb[2]).astype(np.float32)
    z = I.project(xb[2:3], w, mu)
    assert np.all(z == 0)


def test_project_orthonormal_basis_keeps_lengths_and_angles():
    """With a full orthonormal basis (v = d) the PCA coordinates are a
    rotation: lengths and inner products of centred rows are preserved."""
    rng = np.random.default_rng(13)
    d = 96
    x = synth.gaussian_rows_f32(10, d, seed=13).to(torch.bfloat16)
    xb = _bits(x)
    w = np.linalg.qr(rng.standard_normal((d, d)))[0].T
    mu = 0.2 * rng.standard_normal(d)
    y = I.project(xb, w, mu, normalize=False)
    xc = O.bf16_bits_to_f64(xb) - mu
    np.testing.assert_allclose(np.linalg.norm(y, axis=1), np.linalg.norm(xc, axis=1), rtol=1e-12)
    np.testing.assert_allclose(y[0] @ y[1], xc[0] @ xc[1], rtol=1e-10)


def test_project_normalised_rows_and_translation():
    rng = np.random.default_rng(14)
    x = synth.gaussian_rows_f32(20, 128, seed=14).to(torch.bfloat16)
    xb = _bits(x)
    w = rng.standard_normal((16, 128)) / np.sqrt(128)
    mu = 0.1 * rng.standard_normal(128)
    y = I.project(xb, w, mu, normalize=False)
    # centring is a translation of the PCA coordinates by -W mu
    np.testing.assert_allclose(y, I.project(xb, w, normalize=False) - w @ mu, atol=1e-12)
    yn = I.project(xb, w, mu)
    np.testing.assert_allclose(np.linalg.norm(yn, axis=1), 1.0, atol=1e-14)
    # the normalised row points along y: positive multiple, and a scaled
    # basis (c > 0) gives the same unit rows
    cos = (yn * y).sum(1) / np.linalg.norm(y, axis=1)
    np.testing.assert_allclose(cos, 1.0, atol=1e-14)
    np.testing.assert_allclose(I.project(xb, 3.0 * w, mu), yn, atol=1e-14)


# ---------------------------------------------------------------- k-means

def test_kmeans_step_bruteforce_and_exact_means():
    rng = np.random.default_rng(5)
    x = _unit(rng, 300, 8)
    init = x[:7].copy()
    for spherical in (True, False):
        a = I.assign_ip(x, init) if spherical else I.assign_l2(x, init)
        xd, cd = x.astype(np.float64), init.astype(np.float64)
        sc = xd @ cd.T if spherical else -((xd[:, None, :] - cd[None]) ** 2).sum(-1)
        best = sc.max(1)
        srt = np.sort(sc, axis=1)
        clear = (srt[:, -1] - srt[:, -2]) > 1e-5
        np.testing.assert_array_equal(a[clear], np.argmax(sc, 1)[clear])
        assert np.all(sc[np.arange(len(x)), a] >= best - 1e-5)
        c, cnt = I.kmeans_update(x, a, init, spherical=False)
        for j in range(7):
            if cnt[j]:
                np.testing.assert_allclose(c[j], xd[a == j].mean(0), atol=2 ** -30 + 1e-7)
            else:
                np.testing.assert_array_equal(c[j], init[j])


def test_kmeans_objective_monotone():
    rng = np.random.default_rng(6)
    x = _unit(rng, 400, 6)
    c = x[:10].copy()
    prev = np.inf
    for _ in range(8):
        a = I.assign_l2(x, c)
        obj = ((x.astype(np.float64) - c[a]) ** 2).sum()
        assert obj <= prev + 1e-9
        prev = obj
        c, _ = I.kmeans_update(x, a, c, spherical=False)
    # spherical: the total inner product to the assigned centroid never drops
    c = I.kmeans(x, x[:10], 1, spherical=True)[0]
    prev = -np.inf
    for _ in range(6):
        a = I.assign_ip(x, c)
        obj = (x.astype(np.float64) * c[a]).sum()
        assert obj >= prev - 1e-9
        prev = obj
        c, _ = I.kmeans_update(x, a, c, spherical=True)


def test_kmeans_separated_clusters_closed_form():
    # four tight groups around +-e0, +-e1: one round from one seed per group
    # gives the group means (and then stays there)
    rng = np.random.default_rng(7)
    base = np.array([[1, 0], [-1, 0], [0, 1], [0, -1]], np.float32)
    lab = rng.integers(0, 4, 200)
    x = (base[lab] + rng.uniform(-0.05, 0.05, (200, 2))).astype(np.float32)
    seeds = np.array([np.nonzero(lab == g)[0][0] for g in range(4)])
    c, a = I.kmeans(x, x[seeds], 3, spherical=False)
    np.testing.assert_array_equal(a, lab)
    for g in range(4):
        np.testing.assert_allclose(c[g], x[lab == g].astype(np.float64).mean(0), atol=1e-7)


# ---------------------------------------------------------------- IVF

def test_ivf_golden():
    g = json.load(open(os.path.join(GOLDEN, "ivf_small.json")))
    x = np.array(g["vectors"], np.float32)
    c = np.array(g["centroids"], np.float32)
    cb = np.array(g["codebooks"], np.float32)
    flat = I.ivf_build(x, c)
    assert flat["cell"].tolist() == g["cell"]
    assert flat["offsets"].tolist() == g["offsets"]
    assert flat["ids"].tolist() == g["ids"]
    q = np.array([g["query"]], np.float32)
    for key, nprobe in (("flat_nprobe1_k2", 1), ("flat_nprobe2_k3", 2), ("flat_nprobe1_k4", 1)):
        k = len(g[key]["idx"])
        s, i, _ = I.ivf_search(flat, c, q, nprobe, k)
        assert i[0].tolist() == g[key]["idx"]
        if "scores" in g[key]:
            assert s[0].tolist() == g[key]["scores"]
    assert s[0, 3] == -np.inf
    pq = I.ivf_build(x, c, cb)
    assert pq["codes"].tolist() == g["codes_list_order"]
    s, i, probes = I.ivf_search(pq, c, q, 2, 4, codebooks=cb)
    assert i[0].tolist() == g["pq_nprobe2_k4"]["idx"]
    assert s[0].tolist() == g["pq_nprobe2_k4"]["scores"]
    assert probes[0].tolist() == [1, 0]


def _index_case(seed, n=600, v=16, nlist=12):
    rng = np.random.default_rng(seed)
    x = _unit(rng, n, v)
    c = I.kmeans(x, x[:nlist], 4, spherical=True)[0]
    return rng, x, c


def test_ivf_build_invariants():
    rng, x, c = _index_case(8)
    ix = I.ivf_build(x, c)
    off, ids = ix["offsets"], ix["ids"]
    assert sorted(ids.tolist()) == list(range(len(x)))
    for cell in range(len(c)):
        mem = ids[off[cell]:off[cell + 1]]
        assert np.all(np.diff(mem) > 0)
        assert np.all(ix["cell"][mem] == cell)
    sc = x.astype(np.float64) @ c.astype(np.float64).T
    srt = np.sort(sc, 1)
    clear = srt[:, -1] - srt[:, -2] > 1e-5
    np.testing.assert_array_equal(ix["cell"][clear], sc.argmax(1)[clear])
    np.testing.assert_array_equal(ix["vectors"], x[ids])


def test_ivf_flat_full_probe_is_exhaustive_search():
    rng, x, c = _index_case(9)
    ix = I.ivf_build(x, c)
    q = _unit(rng, 5, x.shape[1])
    s, i, _ = I.ivf_search(ix, c, q, len(c), 20)
    ex = q.astype(np.float64) @ x.astype(np.float64).T
    for qi in range(5):
        o = np.lexsort((np.arange(len(x)), -ex[qi]))[:20]
        kth = ex[qi, o[-1]]
        for r in set(i[qi].tolist()) ^ set(o.tolist()):
            assert abs(ex[qi, r] - kth) < 1e-5
        np.testing.assert_allclose(s[qi], ex[qi, i[qi]], atol=1e-5)


def test_ivf_probes_are_top_cells_and_results_come_from_them():
    rng, x, c = _index_case(10)
    ix = I.ivf_build(x, c)
    q = _unit(rng, 6, x.shape[1])
    s, i, probes = I.ivf_search(ix, c, q, 3, 10)
    cs = q.astype(np.float64) @ c.astype(np.float64).T
    for qi in range(6):
        third = np.sort(cs[qi])[-3]
        assert np.all(cs[qi, probes[qi]] >= third - 1e-6)
        assert set(ix["cell"][i[qi]].tolist()) <= set(probes[qi].tolist())


def test_ivf_pq_exact_codebooks_reduce_to_flat():
    # residual sub-vectors take few distinct values, all present in the
    # codebooks: PQ decoding is exact, so IVF-PQ scores are the flat scores
    rng = np.random.default_rng(11)
    v, pq_m, nlist, n = 8, 4, 3, 300
    dsub = v // pq_m
    c = np.zeros((nlist, v), np.float32)
    c[np.arange(nlist), np.arange(nlist)] = 1.0
    vals = (rng.integers(-4, 5, (pq_m, 256, dsub)) / 8).astype(np.float32)
    codes = rng.integers(0, 256, (n, pq_m))
    cell = rng.integers(0, nlist, n)
    r = np.concatenate([vals[m][codes[:, m]] for m in range(pq_m)], axis=1)
    x = (c[cell] + r).astype(np.float32)
    ix = I.ivf_build(x, c, vals)
    # decoded vectors equal the vectors (codes may differ only between equal codewords)
    inv = np.empty(n, np.int64)
    inv[ix["ids"]] = np.arange(n)
    dec = np.concatenate([vals[m][ix["codes"][inv, m]] for m in range(pq_m)], axis=1)
    np.testing.assert_array_equal(dec + c[ix["cell"]], x)
    q = (rng.integers(-4, 5, (4, v)) / 8).astype(np.float32)
    flat = I.ivf_build(x, c)
    s1, i1, _ = I.ivf_search(flat, c, q, nlist, 25)
    s2, i2, _ = I.ivf_search(ix, c, q, nlist, 25, codebooks=vals)
    np.testing.assert_array_equal(s1, s2)
    np.testing.assert_array_equal(i1, i2)


def test_recall_at_k():
    assert I.recall_at_k(np.array([[1, 2, 3]]), np.array([[3, 4, 1]])) == pytest.approx(2 / 3)


# ---------------------------------------------------------------- shortlist re-scoring (Eq. 8 sim)

def test_rescore_topk_exact_on_lattice_and_ordering():
    """Lattice keys make every score an exact short binary fraction: the
    re-scored top k must equal brute force with rational arithmetic, ties
    broken by the lower key index, empty slots (-1) skipped and padded."""
    from fractions import Fraction as F
    rng = np.random.default_rng(21)
    n, d = 40, 16
    kv = rng.integers(-3, 4, (n, d)) / 64.0
    qv = rng.integers(-3, 4, (3, d)) / 64.0
    kb = _bits(torch.tensor(kv, dtype=torch.float32).to(torch.bfloat16))
    qb = _bits(torch.tensor(qv, dtype=torch.float32).to(torch.bfloat16))
    cand = np.array([rng.permutation(n)[:12], np.r_[rng.permutation(n)[:5], [-1] * 7],
                     np.r_[[-1] * 10, [3, 17]]], dtype=np.int32)
    for k in (1, 4, 8):
        s, i = I.rescore_topk(kb, qb, cand, k)
        for qi in range(3):
            c = [int(x) for x in cand[qi] if x >= 0]
            ex = sorted(((sum(F(float(qv[qi, j])) * F(float(kv[r, j])) for j in range(d)), r)
                         for r in c), key=lambda t: (-t[0], t[1]))[:k]
            assert [r for _, r in ex] == i[qi, :len(ex)].tolist()
            assert [float(v) for v, _ in ex] == s[qi, :len(ex)].tolist()
            assert np.all(i[qi, len(ex):] == -1) and np.all(s[qi, len(ex):] == -np.inf)


def test_rescore_of_every_key_is_exhaustive_search():
    # a shortlist holding every key reduces to the exact top-k of the store
    rng = np.random.default_rng(22)
    x = synth.gaussian_rows_f32(300, 32, seed=22).to(torch.bfloat16)
    q = synth.gaussian_rows_f32(2, 32, seed=23).to(torch.bfloat16)
    kb, qb = _bits(x), _bits(q)
    cand = np.stack([rng.permutation(300) for _ in range(2)]).astype(np.int32)
    s, i = I.rescore_topk(kb, qb, cand, 25)
    full = O.bf16_bits_to_f64(qb) @ O.bf16_bits_to_f64(kb).T
    for qi in range(2):
        o = np.lexsort((np.arange(300), -full[qi]))[:25]
        assert i[qi].tolist() == o.tolist()
        np.testing.assert_allclose(s[qi], full[qi, o], rtol=0, atol=1e-12)
