"""GPU-vs-oracle parity of the approximate retrieval path (PCA projection,
k-means, IVF-flat / IVF-PQ build and search), through the C ABI.

The projection is compared with the oracle's fp64 definition within the
error bound of fp32 arithmetic (``_projection_bound``).  Every later step
ends in an integer decision that both sides take in fp32 on the SAME input
vectors (the tests hand the oracle the GPU's projected vectors where a
chain starts from hidden states), summing projected-space products left to
right, so those outputs are compared bit for bit: centroids, assignments,
lists, codes, probes, scores and indices.  Inputs come from seeded
generators; expected values only from ``oracle``.
"""
import json
import os

import numpy as np
import pytest
import torch

import synth
from oracle import ivf_oracle as I
from tests.parity import bits, host

pytestmark = pytest.mark.gpu
cuda = pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(scope="module")
def S():
    import paper_2606_00021_gb300 as S
    S.lib()
    return S


def _unit(rng, n, d):
    x = rng.standard_normal((n, d))
    return (x / np.linalg.norm(x, axis=1, keepdims=True)).astype(np.float32)


def _clustered(rng, n, v, nclust, spread=0.25):
    c = _unit(rng, nclust, v)
    x = c[rng.integers(0, nclust, n)] + spread / np.sqrt(v) * rng.standard_normal((n, v))
    return (x / np.linalg.norm(x, axis=1, keepdims=True)).astype(np.float32)


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


# ---------------------------------------------------------------- projection

U32 = 2.0 ** -24  # fp32 unit roundoff


def _projection_bound(x_bits, w, mu, normalize):
    """Largest |fp32 result - exact result| per element of the projection.

    Unnormalised: the library rounds each centred value (x_j - mu_j) once and
    each product once, and adds the d products in a tree whose every term
    passes through at most h = 4 ceil(d / 128) + 5 additions (32 partial
    sums of 4-column groups, then 5 rounds combining them), so
    |error| <= (h + 2) u sum_j |x_j - mu_j| |w_oj| to first order
    (u = 2^-24; 1% added for the higher-order terms).
    Normalised: with e the error of y and b its bound,
    |(y + e)_i / ||y + e|| - y_i / ||y|| | <= (b_i + |y_i| ||b|| / ||y||) /
    (||y|| - ||b||), and the fp32 norm (v squares summed, a square root, a
    division) adds at most (v + 4) u to each unit entry."""
    x = I.bf16_bits_to_f64(x_bits)
    w = np.asarray(w, np.float64)
    xc = x - (0.0 if mu is None else np.asarray(mu, np.float64)[None, :])
    d, v = x.shape[1], w.shape[0]
    h = 4 * ((d + 127) // 128) + 5
    b = 1.01 * (h + 2) * U32 * (np.abs(xc) @ np.abs(w).T)
    if not normalize:
        return b
    y = xc @ w.T
    ny = np.linalg.norm(y, axis=1, keepdims=True)
    nb = np.linalg.norm(b, axis=1, keepdims=True)
    assert np.all(nb < 0.5 * ny)
    return (b + np.abs(y) * nb / ny) / (ny - nb) + (v + 4) * U32


@cuda
@pytest.mark.parametrize("n,d,v,centre,norm", [
    (1, 4096, 64, True, True), (5, 1000, 16, False, True), (300, 4096, 64, True, True),
    (333, 1000, 48, True, False), (40, 512, 128, False, True), (2000, 256, 20, True, True),
    (3, 768, 20, True, False), (64, 4096, 64, True, True), (2, 2048, 60, True, True),
    (129, 8192, 64, True, True), (17, 3584, 64, True, False),
])
def test_project_matches_oracle(S, n, d, v, centre, norm):
    rng = np.random.default_rng(n + d + v)
    x = synth.gaussian_rows_f32(n, d, seed=n).to(torch.bfloat16)
    w = (rng.standard_normal((v, d)) / np.sqrt(d)).astype(np.float32)
    mu = (0.1 * rng.standard_normal(d)).astype(np.float32) if centre else None
    got = S.sense_project(x.cuda(), _dev(w), None if mu is None else _dev(mu), normalize=norm)
    torch.cuda.synchronize()
    xb = bits(x)
    want = I.project(xb, w, mu, normalize=norm)
    err = np.abs(host(got).astype(np.float64) - want)
    bound = _projection_bound(xb, w, mu, norm)
    assert np.all(err <= bound), f"projection error {err.max():.3g} above its bound"
    # the bound means something: dropping the largest term of a sum
    # (or flipping its sign) would leave it
    xc = I.bf16_bits_to_f64(xb) - (0.0 if mu is None else mu.astype(np.float64))
    biggest = np.abs(xc)[:, None, :] * np.abs(w.astype(np.float64))[None, :, :]
    term = biggest.max(axis=2)
    if norm:
        term = term / np.linalg.norm(xc @ w.astype(np.float64).T, axis=1, keepdims=True)
    assert np.mean(term > bound) > 0.9


# ---------------------------------------------------------------- k-means

@cuda
@pytest.mark.parametrize("n,dim,ld,k,iters,sph", [
    (2000, 64, 64, 16, 3, True), (3000, 16, 16, 256, 2, False), (1500, 4, 64, 256, 3, False),
    (500, 32, 32, 7, 0, True), (4100, 128, 128, 40, 2, True),
])
def test_kmeans_matches_oracle(S, n, dim, ld, k, iters, sph):
    rng = np.random.default_rng(n + k)
    x = _clustered(rng, n, ld, 12) if ld >= 16 else rng.standard_normal((n, ld)).astype(np.float32)
    init = x[rng.choice(n, size=k, replace=False), :dim].copy()
    cent, assign = S.sense_kmeans(_dev(x)[:, :dim], _dev(init), iters, sph, want_assign=True)
    torch.cuda.synchronize()
    want_c, want_a = I.kmeans(x[:, :dim], init, iters, sph)
    np.testing.assert_array_equal(host(cent), want_c)
    if iters:
        np.testing.assert_array_equal(host(assign), want_a)


# ---------------------------------------------------------------- index build

def _index_inputs(seed, n, v, nlist, pq_m):
    rng = np.random.default_rng(seed)
    x = _clustered(rng, n, v, max(4, nlist // 2))
    cent = _unit(rng, nlist, v)
    cb = None
    if pq_m:
        dsub = v // pq_m
        cb = (0.3 / np.sqrt(v) * rng.standard_normal((pq_m, 256, dsub))).astype(np.float32)
    return rng, x, cent, cb


@cuda
@pytest.mark.parametrize("n,v,nlist,pq_m", [
    (5000, 64, 64, 0), (5000, 64, 64, 16), (9000, 16, 300, 4), (1, 32, 8, 8), (700, 128, 9, 8),
])
def test_ivf_build_matches_oracle(S, n, v, nlist, pq_m):
    _, x, cent, cb = _index_inputs(n + nlist, n, v, nlist, pq_m)
    ix = S.sense_ivf_build(_dev(x), _dev(cent), None if cb is None else _dev(cb))
    arr = ix.arrays()
    torch.cuda.synchronize()
    want = I.ivf_build(x, cent, cb)
    np.testing.assert_array_equal(host(arr["offsets"]), want["offsets"])
    np.testing.assert_array_equal(host(arr["ids"]), want["ids"])
    assert ix.max_list == int(np.diff(want["offsets"]).max())
    if pq_m:
        np.testing.assert_array_equal(host(arr["codes"]), want["codes"])
    else:
        np.testing.assert_array_equal(host(arr["vectors"]), want["vectors"])
    cell, res = S.sense_ivf_residuals(_dev(x), _dev(cent))
    torch.cuda.synchronize()
    np.testing.assert_array_equal(host(cell), want["cell"])
    np.testing.assert_array_equal(host(res), x - cent[want["cell"]])
    ix.close()


# ---------------------------------------------------------------- search

@cuda
@pytest.mark.parametrize("n,v,nlist,pq_m,q,k,nprobe", [
    (6000, 64, 64, 0, 1, 32, 8), (6000, 64, 64, 16, 7, 100, 8), (6000, 64, 64, 16, 64, 16, 64),
    (9000, 16, 300, 4, 5, 64, 1), (3000, 32, 40, 0, 33, 256, 3), (2000, 64, 16, 16, 3, 500, 2),
    (20000, 64, 64, 16, 4, 512, 16), (12000, 32, 64, 16, 3, 300, 32), (20000, 64, 64, 0, 2, 1024, 64),
])
def test_ivf_search_matches_oracle(S, n, v, nlist, pq_m, q, k, nprobe):
    """Probes, indices and scores bit-identical to the oracle's search: the
    pool merge's short path (k below the number of 32-key groups), its
    binned path (larger k), the radix path (a pool too long for the binned
    path's shared memory) and short pools padded with -inf / -1."""
    rng, x, cent, cb = _index_inputs(7 * n + q, n, v, nlist, pq_m)
    qs = _clustered(rng, q, v, 8)
    ix = S.sense_ivf_build(_dev(x), _dev(cent), None if cb is None else _dev(cb))
    sc, idx, probes = S.sense_ivf_search(ix, _dev(qs), k, nprobe, want_probes=True)
    torch.cuda.synchronize()
    assert S.sense_device_status(clear=True) == 0
    index = I.ivf_build(x, cent, cb)
    ws, wi, wp = I.ivf_search(index, cent, qs, nprobe, k, codebooks=cb)
    np.testing.assert_array_equal(host(probes), wp)
    np.testing.assert_array_equal(host(idx), wi)
    np.testing.assert_array_equal(host(sc), ws)
    ix.close()


@cuda
@pytest.mark.parametrize("n,k", [(6000, 600), (3000, 300)])
def test_ivf_search_equal_scores(S, n, k):
    """Every vector identical: every candidate ties, so the top k are the k
    lowest key indices.  Longer pools put more keys in one score bin than
    the binned selection holds and take the radix path (n = 6000); shorter
    ones rank a single bucket (n = 3000)."""
    rng = np.random.default_rng(n)
    v, nlist = 32, 4
    one = _unit(rng, 1, v)
    x = np.repeat(one, n, axis=0).astype(np.float32)
    cent = _unit(rng, nlist, v)
    qs = _unit(rng, 2, v)
    ix = S.sense_ivf_build(_dev(x), _dev(cent))
    sc, idx = S.sense_ivf_search(ix, _dev(qs), k, nlist)
    torch.cuda.synchronize()
    assert S.sense_device_status(clear=True) == 0
    index = I.ivf_build(x, cent, None)
    ws, wi, _ = I.ivf_search(index, cent, qs, nlist, k)
    np.testing.assert_array_equal(host(idx), wi)
    np.testing.assert_array_equal(host(sc), ws)
    assert host(idx)[0].tolist() == list(range(k))
    ix.close()


@cuda
def test_rescore_portable_cluster_width():
    """The re-scoring kernel's portable cluster width (8 CTAs per query,
    used where a cluster of 16 cannot be resident), forced through
    SENSE_RESCORE_CLUSTER in a fresh process: bit-exact on lattice keys at
    shortlists that need 1, 2 and 4 keys per lane in the per-CTA sort."""
    import subprocess
    import sys
    code = r"""
import numpy as np, torch, sys
sys.path.insert(0, '.')
import paper_2606_00021_gb300 as S, synth
from oracle import ivf_oracle as I
from tests.parity import bits, host
dev = torch.device('cuda')
n, d, q = 6000, 512, 2
keys = synth.lattice_rows(n, d, seed=7, device=dev)
qs = synth.lattice_rows(q, d, seed=8, device=dev)
ds = S.sense_datastore_build(keys, synth.spans_uniform(n, 2, 50, seed=1, device=dev))
rng = np.random.default_rng(3)
for n_cand, k in ((200, 50), (500, 100), (1024, 1024)):
    cand = np.stack([rng.permutation(n)[:n_cand] for _ in range(q)]).astype(np.int32)
    sc, ix = S.sense_rescore_topk(ds, qs, torch.from_numpy(cand).to(dev), k)
    torch.cuda.synchronize()
    assert S.sense_device_status(clear=True) == 0
    ws, wi = I.rescore_topk(bits(keys), bits(qs), cand, k)
    np.testing.assert_array_equal(host(ix), wi)
    np.testing.assert_array_equal(host(sc).astype(np.float64), ws)
print('ok')
"""
    env = dict(__import__("os").environ, SENSE_RESCORE_CLUSTER="8")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env,
                       cwd=os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                       timeout=600)
    assert r.returncode == 0 and r.stdout.strip().endswith("ok"), r.stderr[-3000:]


@cuda
def test_ivf_golden_on_gpu(S):
    """The hand-worked index, embedded in 16 dimensions: the extra
    coordinates are zero, their codebooks code zero first, and the golden
    codebooks fill codewords 0..3 of sub-quantizers 0 and 1 (the rest lie
    far away)."""
    g = json.load(open(os.path.join(GOLDEN, "ivf_small.json")))
    v, pq_m = 16, 16
    x = np.zeros((5, v), np.float32)
    x[:, :2] = g["vectors"]
    c = np.zeros((2, v), np.float32)
    c[:, :2] = g["centroids"]
    cb = np.full((pq_m, 256, 1), 1000.0, np.float32)
    cb[2:, 0, 0] = 0.0
    for m in range(2):
        cb[m, :4, 0] = np.array(g["codebooks"][m])[:, 0]
    ixf = S.sense_ivf_build(_dev(x), _dev(c))
    ixp = S.sense_ivf_build(_dev(x), _dev(c), _dev(cb))
    qv = np.zeros((1, v), np.float32)
    qv[0, :2] = g["query"]
    arr = ixp.arrays()
    assert host(arr["ids"]).tolist() == g["ids"]
    assert host(arr["codes"])[:, :2].tolist() == g["codes_list_order"]
    s, i = S.sense_ivf_search(ixf, _dev(qv), 3, 2)
    assert host(i)[0].tolist() == g["flat_nprobe2_k3"]["idx"]
    assert host(s)[0].tolist() == g["flat_nprobe2_k3"]["scores"]
    s, i = S.sense_ivf_search(ixf, _dev(qv), 4, 1)
    assert host(i)[0].tolist() == g["flat_nprobe1_k4"]["idx"]
    assert host(s)[0, 3] == -np.inf
    s, i = S.sense_ivf_search(ixp, _dev(qv), 4, 2)
    assert host(i)[0].tolist() == g["pq_nprobe2_k4"]["idx"]
    assert host(s)[0].tolist() == g["pq_nprobe2_k4"]["scores"]
    assert S.sense_device_status(clear=True) == 0


@cuda
def test_projected_pipeline_and_recall(S):
    """Hidden states -> PCA-64 keys -> k-means cells -> IVF-PQ, all on the
    GPU.  The projected keys and queries are within the fp32 bound of the
    oracle's exact projection; from them on, the oracle's chain runs on the
    GPU's projected vectors (the same inputs as the GPU's chain) and must
    agree bit for bit (the k-means seeds are rows of those vectors and
    residuals).  Recall@k of IVF-flat against the exact search in the
    projected space is high when most cells are probed."""
    rng = np.random.default_rng(99)
    n, d, v, nlist, pq_m, q, k = 6000, 1024, 64, 32, 16, 6, 20
    keys = synth.clustered_unit_keys(n, d, 24, seed=3)
    qh, _ = synth.noisy_queries(keys, q, seed=4)
    w = np.linalg.qr(rng.standard_normal((d, v)))[0].T.astype(np.float32).copy()
    kp = S.sense_project(keys.cuda(), _dev(w))
    qp = S.sense_project(qh.cuda(), _dev(w))
    torch.cuda.synchronize()
    kp_h, qp_h = host(kp), host(qp)
    for xb, got in ((bits(keys), kp_h), (bits(qh), qp_h)):
        err = np.abs(got.astype(np.float64) - I.project(xb, w))
        assert np.all(err <= _projection_bound(xb, w, None, True))
    init = kp_h[rng.choice(n, nlist, replace=False)].copy()
    # oracle chain on the GPU's projected vectors
    cent_w = I.kmeans(kp_h, init, 4, True)[0]
    res_w = kp_h - cent_w[I.assign_ip(kp_h, cent_w)]
    cb_init = np.stack([res_w[:256, m * 4:(m + 1) * 4] for m in range(pq_m)])
    cb_w = np.stack([I.kmeans(res_w[:, m * 4:(m + 1) * 4], cb_init[m], 3, False)[0]
                     for m in range(pq_m)])
    ws, wi, _ = I.ivf_search(I.ivf_build(kp_h, cent_w, cb_w), cent_w, qp_h, 8, k, codebooks=cb_w)
    # GPU chain from the same vectors
    cent = S.sense_kmeans(kp, _dev(init), 4, True)
    cell, res = S.sense_ivf_residuals(kp, cent)
    # sub-quantizer m trains on columns 4m..4m+3 of the residuals (row stride v)
    cbs = [S.sense_kmeans(res[:, 4 * m:4 * m + 4], _dev(cb_init[m]), 3, False)
           for m in range(pq_m)]
    ix = S.sense_ivf_build(kp, cent, torch.stack(cbs))
    sc, idx = S.sense_ivf_search(ix, qp, k, 8)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(host(cent), cent_w)
    np.testing.assert_array_equal(host(res), res_w)
    np.testing.assert_array_equal(host(torch.stack(cbs)), cb_w)
    np.testing.assert_array_equal(host(idx), wi)
    np.testing.assert_array_equal(host(sc), ws)
    flat = S.sense_ivf_build(kp, cent)
    _, fi = S.sense_ivf_search(flat, qp, k, 24)
    exact = np.argsort(-(qp_h.astype(np.float64) @ kp_h.astype(np.float64).T), axis=1)[:, :k]
    assert I.recall_at_k(host(fi), exact) > 0.9


# ---------------------------------------------------------------- shortlist re-scoring (Eq. 8 sim)

@cuda
@pytest.mark.parametrize("n,d,q,n_cand,k,empty", [
    (50000, 512, 5, 300, 32, 0), (20000, 4096, 3, 1024, 64, 100), (9000, 256, 2, 1, 1, 0),
    (9000, 256, 4, 40, 40, 30), (70000, 8192, 1, 256, 32, 0), (5000, 4104, 2, 600, 50, 20),
    (8000, 4096, 1, 512, 32, 0), (8000, 4096, 1, 513, 32, 0), (3000, 64, 2, 1000, 999, 5),
])
def test_rescore_matches_oracle(S, n, d, q, n_cand, k, empty):
    """Exact re-scoring of a shortlist: scores within 2e-3 of the oracle's
    fp64 inner products, the top-k rule of the exact search restricted to
    the candidates, and empty slots (-1) skipped and padded with -inf / -1."""
    from tests.parity import check_topk
    dev = torch.device("cuda")
    rng = np.random.default_rng(n + n_cand)
    keys = synth.clustered_unit_keys(n, d, 64, seed=n % 97, device=dev)
    qs, _ = synth.noisy_queries(keys, q, seed=5)
    ds = S.sense_datastore_build(keys, synth.spans_uniform(n, 2, 50, seed=1, device=dev))
    cand = np.stack([rng.permutation(n)[:n_cand] for _ in range(q)]).astype(np.int32)
    for qi in range(q):
        cand[qi, rng.permutation(n_cand)[:empty]] = -1
    sc, ix = S.sense_rescore_topk(ds, qs, _dev(cand), k)
    torch.cuda.synchronize()
    assert S.sense_device_status(clear=True) == 0
    ws, wi = I.rescore_topk(bits(keys), bits(qs), cand, k)
    for qi in range(q):
        valid = int((wi[qi] >= 0).sum())
        assert host(ix[qi])[valid:].tolist() == [-1] * (k - valid)
        assert np.all(host(sc[qi])[valid:] == -np.inf)
        row = np.full(n, -np.inf)
        c = cand[qi][cand[qi] >= 0]
        row[c] = I.scores(bits(keys)[c], bits(qs[qi:qi + 1]))[0]
        check_topk(host(sc[qi])[:valid], host(ix[qi])[:valid], row, valid)


@cuda
@pytest.mark.parametrize("d,n_cand,k,dup", [(512, 500, 100, 0), (512, 1024, 1024, 40),
                                             (8200, 17, 5, 3), (512, 64, 64, 0)])
def test_rescore_lattice_bit_exact_and_bad_index(S, d, n_cand, k, dup):
    """Lattice keys and queries: every score is exact in fp32, so scores,
    order and ties (lower key index first) must equal the oracle bit for
    bit, at the largest shortlist and with repeated candidates (each copy
    is scored and kept).  An index outside [0, n) is skipped and reported."""
    dev = torch.device("cuda")
    n, q = 6000, 3
    keys = synth.lattice_rows(n, d, seed=7, device=dev)
    qs = synth.lattice_rows(q, d, seed=8, device=dev)
    ds = S.sense_datastore_build(keys, synth.spans_uniform(n, 2, 50, seed=1, device=dev))
    rng = np.random.default_rng(3)
    cand = np.stack([rng.permutation(n)[:n_cand] for _ in range(q)]).astype(np.int32)
    if dup:
        cand[:, :dup] = cand[:, n_cand - dup:]
    sc, ix = S.sense_rescore_topk(ds, qs, _dev(cand), k)
    torch.cuda.synchronize()
    assert S.sense_device_status(clear=True) == 0
    ws, wi = I.rescore_topk(bits(keys), bits(qs), cand, k)
    np.testing.assert_array_equal(host(ix), wi)
    np.testing.assert_array_equal(host(sc).astype(np.float64), ws)
    bad = cand.copy()
    bad[0, 7] = n + 5
    bad[1, 0] = 1 << 30
    sc2, ix2 = S.sense_rescore_topk(ds, qs, _dev(bad), k)
    torch.cuda.synchronize()
    assert S.sense_device_status(clear=True) == S.DEVST_BAD_INDEX
    bad[bad >= n] = -1
    ws2, wi2 = I.rescore_topk(bits(keys), bits(qs), bad, k)
    np.testing.assert_array_equal(host(ix2), wi2)


# ---------------------------------------------------------------- approximate drafting step in one call

@cuda
@pytest.mark.parametrize("pq,rerank,q,k,cap,nlist,nprobe", [
    (False, 0, 1, 32, 64, 64, 8), (True, 0, 1, 32, 64, 64, 8), (True, 128, 1, 32, 64, 64, 8),
    (True, 64, 3, 16, 0, 64, 8), (False, 40, 2, 40, 30, 64, 8),
    (True, 0, 2, 200, 64, 64, 8), (True, 300, 1, 200, 0, 64, 8),
    (False, 0, 2, 128, 64, 1024, 1), (True, 0, 1, 100, 0, 1024, 1),
])
def test_ann_draft_equals_separate_calls(S, pq, rerank, q, k, cap, nlist, nprobe):
    """sense_ann_draft is bit-identical to projection, IVF search (and the
    exact re-scoring), gather and trie called one by one: with the fused
    tails (k <= 128), without them (k = 200), and with a probed list shorter
    than k (the pool is padded with -inf / -1)."""
    dev = torch.device("cuda")
    rng = np.random.default_rng(17 + k)
    n, d, v = 20000, 512, 32
    keys = synth.clustered_unit_keys(n, d, 32, seed=19, device=dev)
    spans = synth.spans_uniform(n, 8, 5, seed=2, device=dev)
    ds = S.sense_datastore_build(keys, spans)
    basis = _dev(np.linalg.qr(rng.standard_normal((d, v)))[0].T.astype(np.float32).copy())
    mean = _dev((0.01 * rng.standard_normal(d)).astype(np.float32))
    kp = S.sense_project(keys, basis, mean)
    cent = S.sense_kmeans(kp[:4096].contiguous(), kp[:nlist].clone(), 3, True)
    cb = None
    if pq:
        _, res = S.sense_ivf_residuals(kp[:4096].contiguous(), cent)
        cb = torch.stack([S.sense_kmeans(res[:, 4 * mm:4 * mm + 4].contiguous(),
                                         res[:256, 4 * mm:4 * mm + 4].contiguous(), 3, False)
                          for mm in range(v // 4)])
    ix = S.sense_ivf_build(kp, cent, cb)
    qs, _ = synth.noisy_queries(keys, q, seed=23)
    for _ in range(2):
        got = S.sense_ann_draft(ix, ds, qs, basis, mean, k, nprobe, rerank=rerank, node_cap=cap,
                                mask_bits=True)
        torch.cuda.synchronize()
        st_one = S.sense_device_status(clear=True)
        qp = S.sense_project(qs, basis, mean)
        if rerank:
            _, ci = S.sense_ivf_search(ix, qp, rerank, nprobe)
            sc, idx = S.sense_rescore_topk(ds, qs, ci, k)
        else:
            sc, idx = S.sense_ivf_search(ix, qp, k, nprobe)
        dr = S.sense_gather_drafts(ds, idx)
        tr = S.sense_build_tree(dr, node_cap=cap, mask_bits=True)
        torch.cuda.synchronize()
        # the same status as the composed calls: none, or for a short pool
        # the -1 slots' rows (bad index, then negative tokens in the trie)
        assert S.sense_device_status(clear=True) == st_one
        assert torch.equal(got["scores"], sc) and torch.equal(got["idx"], idx)
        sc2, ix2 = S.sense_ann_search(ix, ds, qs, basis, mean, k, nprobe, rerank=rerank)
        torch.cuda.synchronize()
        assert torch.equal(sc2, sc) and torch.equal(ix2, idx)
        if nprobe > 1:
            assert S.sense_device_status(clear=True) == 0
        else:
            S.sense_device_status(clear=True)
        if nprobe == 1:  # a short pool: the padding is part of the result
            assert (idx == -1).any()
            assert st_one == S.DEVST_BAD_INDEX | S.DEVST_BAD_TOKEN
        else:
            assert st_one == 0
        assert torch.equal(got["spans"], dr)
        for key in ("num_nodes", "tokens", "parent", "depth", "gamma", "mask_bits"):
            assert torch.equal(got[key], tr[key]), key
    ix.close()


@cuda
@pytest.mark.parametrize("v,nlist,nprobe,pq", [
    (64, 2048, 33, False),   # one 256-cell tile per block of the 8-block cluster
    (64, 4096, 64, True),    # two tiles per block
    (64, 6144, 17, False),   # three tiles per block
    (64, 8192, 64, False),   # four tiles per block
    (64, 4096, 100, False),
    (16, 4096, 32, False),   # two blocks, eight tiles each
    (64, 4096, 1, False),
])
def test_ann_search_cell_selection(S, v, nlist, nprobe, pq):
    """The query-side launch's cell selection (coarse keys of the cluster's
    blocks merged in block 0's shared memory) probes the same cells as the
    coarse scores and merge called one by one: k = 1024 over short lists
    returns every scanned entry, so equal results mean equal cell sets."""
    dev = torch.device("cuda")
    rng = np.random.default_rng(nlist + nprobe)
    n, d, q, k = 20000, 512, 2, 1024
    keys = synth.clustered_unit_keys(n, d, 64, seed=29, device=dev)
    spans = synth.spans_uniform(n, 8, 5, seed=2, device=dev)
    ds = S.sense_datastore_build(keys, spans)
    basis = _dev(np.linalg.qr(rng.standard_normal((d, v)))[0].T.astype(np.float32).copy())
    mean = _dev((0.01 * rng.standard_normal(d)).astype(np.float32))
    kp = S.sense_project(keys, basis, mean)
    cent = S.sense_kmeans(kp, kp[:nlist].clone(), 2, True)
    cb = None
    if pq:
        _, res = S.sense_ivf_residuals(kp, cent)
        cb = torch.stack([S.sense_kmeans(res[:, 4 * mm:4 * mm + 4].contiguous(),
                                         res[:256, 4 * mm:4 * mm + 4].contiguous(), 2, False)
                          for mm in range(v // 4)])
    ix = S.sense_ivf_build(kp, cent, cb)
    qs, _ = synth.noisy_queries(keys, q, seed=31)
    sc, idx = S.sense_ann_search(ix, ds, qs, basis, mean, k, nprobe)
    torch.cuda.synchronize()
    st_one = S.sense_device_status(clear=True)
    qp = S.sense_project(qs, basis, mean)
    sc2, idx2, probes = S.sense_ivf_search(ix, qp, k, nprobe, want_probes=True)
    torch.cuda.synchronize()
    assert S.sense_device_status(clear=True) == st_one
    sizes = (ix.arrays()["offsets"][1:] - ix.arrays()["offsets"][:-1])
    scanned = sizes[probes.long()].sum(dim=1)
    assert int(scanned.max()) < k  # the whole pool is in the result
    assert torch.equal(sc, sc2) and torch.equal(idx, idx2)
    for qi in range(q):
        got = set(idx[qi][idx[qi] >= 0].tolist())
        assert len(got) == int(scanned[qi])
    ix.close()
