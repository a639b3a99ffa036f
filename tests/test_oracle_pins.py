"""Pins of the CPU oracle to facts fixed by the paper and by mathematics.

Each test checks the oracle against something other than itself: exact
rational arithmetic, closed forms, brute force on tiny inputs, library
routines in special cases, invariants, and hand-worked examples stored under
tests/golden/ (each with its citation).  No GPU is needed.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle as O
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


# --------------------------------------------------------------------------
# bf16 codec
# --------------------------------------------------------------------------

def test_bf16_decode_matches_torch():
    rng = np.random.default_rng(0)
    bits = rng.integers(0, 1 << 16, size=20000, dtype=np.uint32).astype(np.uint16)
    exp = (bits >> 7) & 0xFF
    bits = bits[exp != 0xFF]  # skip inf/nan encodings
    ref = torch.from_numpy(bits.view(np.int16).copy()).view(torch.bfloat16).double().numpy()
    np.testing.assert_array_equal(O.bf16_bits_to_f64(bits), ref)


def test_bf16_round_matches_torch_rne():
    rng = np.random.default_rng(1)
    x = np.concatenate([
        rng.standard_normal(20000).astype(np.float32),
        (rng.standard_normal(2000) * 1e-39).astype(np.float32),  # subnormals
        rng.uniform(-1, 1, 2000).astype(np.float32),
    ])
    # exact halfway cases: low 16 bits == 0x8000 (ties go to even)
    hw = (rng.integers(0x3F000000, 0x40000000, 2000, dtype=np.uint32) & 0xFFFF0000) | 0x8000
    x = np.concatenate([x, hw.view(np.float32)])
    ref = _bits(torch.from_numpy(x).to(torch.bfloat16))
    np.testing.assert_array_equal(O.f64_to_bf16_bits(x.astype(np.float64)), ref)


# --------------------------------------------------------------------------
# a1: normalisation
# --------------------------------------------------------------------------

def test_normalize_unit_norm_and_scale_invariance():
    x = synth.gaussian_rows_f32(64, 4096, seed=3).numpy()
    y = O.normalize_keys_bf16(x)
    yf = O.bf16_bits_to_f64(y)
    norms = np.linalg.norm(yf, axis=1)
    # bf16 relative rounding <= 2^-9 per coordinate
    assert np.all(np.abs(norms - 1.0) < 2.0 ** -8)
    np.testing.assert_array_equal(O.normalize_keys_bf16(x * 8.0), y)
    np.testing.assert_array_equal(O.normalize_keys_bf16(np.zeros((2, 16))), np.zeros((2, 16), np.uint16))


def test_normalize_close_to_torch():
    x = synth.gaussian_rows_f32(32, 512, seed=4)
    ref = _bits(torch.nn.functional.normalize(x.double(), dim=1).to(torch.bfloat16))
    got = O.normalize_keys_bf16(x.numpy())
    # torch rounds fp64 -> bf16 once as well; allow a 1-ulp difference
    diff = np.abs(got.astype(np.int32) - ref.astype(np.int32))
    assert diff.max() <= 1
    assert (diff == 0).mean() > 0.999


# --------------------------------------------------------------------------
# a2: scores
# --------------------------------------------------------------------------

def test_scores_exact_rational_bruteforce():
    keys = synth.clustered_unit_keys(24, 64, 4, seed=5)
    qs, _ = synth.noisy_queries(keys, 3, seed=5)
    kb, qb = _bits(keys), _bits(qs)
    s = O.scores(kb, qb, chunk=7)
    kf, qf = O.bf16_bits_to_f64(kb), O.bf16_bits_to_f64(qb)
    for q in range(3):
        for i in range(24):
            exact = sum(Fraction(float(a)) * Fraction(float(b)) for a, b in zip(qf[q], kf[i]))
            assert abs(Fraction(s[q, i]) - exact) <= Fraction(1, 1 << 50)


def test_scores_lattice_integer_exact():
    keys = synth.lattice_rows(300, 256, seed=6)
    qs = synth.lattice_rows(4, 256, seed=7)
    s = O.scores(_bits(keys), _bits(qs))
    ki = np.rint(keys.float().numpy() * 64).astype(np.int64)
    qi = np.rint(qs.float().numpy() * 64).astype(np.int64)
    exact = (qi @ ki.T).astype(np.float64) * 2.0 ** -12
    np.testing.assert_array_equal(s, exact)


def test_scores_basis_and_self():
    d = 128
    eye = torch.eye(d, dtype=torch.float32).to(torch.bfloat16)
    q = synth.gaussian_rows_f32(2, d, seed=8).to(torch.bfloat16)
    s = O.scores(_bits(eye), _bits(q))
    np.testing.assert_array_equal(s, q.double().numpy())
    keys = synth.clustered_unit_keys(50, 1024, 8, seed=9)
    ss = O.scores(_bits(keys), _bits(keys))
    kf = keys.double().numpy()
    np.testing.assert_allclose(np.diag(ss), np.einsum("ij,ij->i", kf, kf), rtol=0, atol=1e-14)
    # Cauchy-Schwarz: |<a,b>| <= |a||b|
    nrm = np.linalg.norm(kf, axis=1)
    assert np.all(np.abs(ss) <= np.outer(nrm, nrm) + 1e-12)


# --------------------------------------------------------------------------
# a3: top-k
# --------------------------------------------------------------------------

@pytest.mark.parametrize("seed", range(5))
def test_topk_bruteforce_with_ties(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(5, 400))
    s = np.round(rng.standard_normal((3, n)), 1)  # heavy ties
    k = int(rng.integers(1, n + 1))
    v, i = O.topk(s, k)
    for q in range(3):
        ref = sorted(range(n), key=lambda j: (-s[q, j], j))[:k]
        assert list(i[q]) == ref
        assert list(v[q]) == [s[q, j] for j in ref]


def test_topk_all_equal_and_full():
    v, i = O.topk(np.zeros((2, 10)), 4)
    assert (i == np.arange(4)).all()
    s = np.array([[3.0, 1.0, 2.0, 3.0]])
    v, i = O.topk(s, 4)
    assert list(i[0]) == [0, 3, 2, 1]
    with pytest.raises(ValueError):
        O.topk(s, 5)


def test_topk_lattice_ties():
    keys = synth.lattice_rows(2000, 64, seed=10)
    qs = synth.lattice_rows(3, 64, seed=11)
    s = O.scores(_bits(keys), _bits(qs))
    v, i = O.topk(s, 50)
    for q in range(3):
        assert np.all(np.diff(v[q]) <= 0)
        same = np.diff(v[q]) == 0
        assert np.all(np.diff(i[q])[same] > 0)
        assert v[q, -1] >= np.sort(s[q])[-50]


# --------------------------------------------------------------------------
# a4: gather (+ Eq. 8 rerank, Alg. 2 forced anchor)
# --------------------------------------------------------------------------

def test_gather_encodes_index():
    n, m = 100, 5
    spans = (np.arange(n)[:, None] * 10 + np.arange(m)[None, :]).astype(np.int32)
    idx = np.array([[3, 99, 0, 42], [7, -1, 100, 5]])
    out = O.gather_drafts(spans, idx)
    assert out.shape == (2, 4, m)
    for q in range(2):
        for r in range(4):
            if 0 <= idx[q, r] < n:
                assert (out[q, r] // 10 == idx[q, r]).all()
                assert (out[q, r] % 10 == np.arange(m)).all()
            else:
                assert (out[q, r] == -1).all()


def test_gather_rerank_equals_eq8_composite():
    rng = np.random.default_rng(12)
    n, m, k = 200, 4, 16
    spans = rng.integers(0, 5, size=(n, m)).astype(np.int32)
    sims = np.sort(rng.uniform(0.5, 1.0, (3, k)))[:, ::-1]  # retrieval order
    idx = rng.choice(n, size=(3, k), replace=False)
    anchor = rng.integers(0, 5, size=3)
    keep = 9
    out = O.gather_drafts(spans, idx, anchor=anchor, n_keep=keep)
    alpha, beta = 1e6, 1.0
    for q in range(3):
        s_eq8 = alpha * (spans[idx[q], 0] == anchor[q]) + beta * sims[q]
        order = np.argsort(-s_eq8, kind="stable")[:keep]
        np.testing.assert_array_equal(out[q], spans[idx[q][order]])
    forced = O.gather_drafts(spans, idx, anchor=anchor, n_keep=keep, force_anchor=True)
    assert (forced[:, 0, 0] == anchor).all() and (forced[:, keep - 1, 0] == anchor).all()
    np.testing.assert_array_equal(forced[:, 1:keep - 1], out[:, 1:keep - 1])


# --------------------------------------------------------------------------
# a5: loose trie
# --------------------------------------------------------------------------

def test_trie_golden():
    g = json.load(open(os.path.join(GOLDEN, "trie_small.json")))
    spans = np.array(g["spans"])
    r = O.loose_trie(spans, mask_bits=True)
    u = g["uncapped"]
    assert r["num_nodes"][0] == u["num_nodes"]
    for key in ("tokens", "parent", "depth"):
        assert list(r[key][0][:u["num_nodes"]]) == u[key]
    assert r["gamma"][0].tolist() == u["gamma"]
    assert r["mask_bits"][0][:9, 0].tolist() == u["mask_words"]
    t_flat, _, _, _ = O.loose_trie_alg3(spans)
    assert t_flat.tolist() == u["t_flat_eq9"]
    c = g["cap5"]
    r5 = O.loose_trie(spans, node_cap=5)
    assert r5["num_nodes"][0] == c["num_nodes"]
    for key in ("tokens", "parent", "depth"):
        assert list(r5[key][0]) == c[key]
    assert r5["gamma"][0].tolist() == c["gamma"]


def _rand_spans(rng, k, m, vocab):
    base = rng.integers(0, vocab, size=(max(1, k // 3), m))
    rows = base[rng.integers(0, base.shape[0], size=k)].copy()
    # mutate suffixes so that prefixes are shared at random depths
    for r in range(k):
        cut = int(rng.integers(0, m + 1))
        rows[r, cut:] = rng.integers(0, vocab, size=m - cut)
    return rows


@pytest.mark.parametrize("seed", range(8))
def test_trie_matches_alg3_and_bruteforce(seed):
    rng = np.random.default_rng(100 + seed)
    k, m = int(rng.integers(1, 24)), int(rng.integers(1, 7))
    spans = _rand_spans(rng, k, m, 4)
    r = O.loose_trie(spans, mask_bits=True)
    t_flat, gam_sorted, mask, pi = O.loose_trie_alg3(spans)
    nn = r["num_nodes"][0]
    prefixes = {tuple(spans[i, :j + 1]) for i in range(k) for j in range(m)}
    assert nn == len(prefixes) == len(t_flat)
    assert r["tokens"][0][:nn].tolist() == t_flat.tolist()
    gam = np.empty_like(gam_sorted)
    gam[pi] = gam_sorted
    assert r["gamma"][0].tolist() == gam.tolist()
    for n in range(nn):
        for b in range(nn):
            bit = (int(r["mask_bits"][0][n, b // 32]) >> (b % 32)) & 1
            assert bit == mask[n, b]


@pytest.mark.parametrize("seed", range(6))
def test_trie_invariants_and_cap(seed):
    rng = np.random.default_rng(200 + seed)
    k, m = int(rng.integers(2, 30)), int(rng.integers(2, 9))
    spans = _rand_spans(rng, k, m, 3)
    full = O.loose_trie(spans)
    nn = full["num_nodes"][0]
    tok, par, dep, gam = full["tokens"][0], full["parent"][0], full["depth"][0], full["gamma"][0]
    paths = []
    for n in range(nn):
        p, chain = n, []
        while p >= 0:
            chain.append(int(tok[p]))
            p = par[p]
        paths.append(tuple(reversed(chain)))
        assert dep[n] == len(chain) - 1
    assert paths == sorted(paths)  # lexicographic preorder
    for r in range(k):
        for j in range(m):
            assert tok[gam[r, j]] == spans[r, j]
            assert par[gam[r, j]] == (gam[r, j - 1] if j else -1)
    # cap: insert spans in rank order, refuse new nodes once C exist
    cap = int(rng.integers(1, nn + 2))
    capped = O.loose_trie(spans, node_cap=cap)
    kept = set()
    for r in range(k):
        for j in range(m):
            p = tuple(spans[r, :j + 1])
            if p not in kept and len(kept) < cap and (j == 0 or tuple(spans[r, :j]) in kept):
                kept.add(p)
    got = set()
    cn = capped["num_nodes"][0]
    for r in range(k):
        for j in range(m):
            if capped["gamma"][0][r, j] >= 0:
                got.add(tuple(spans[r, :j + 1]))
    assert got == kept and cn == len(kept) == min(cap, nn)


def test_trie_special_cases():
    m = 6
    same = np.tile(np.arange(m), (5, 1))
    assert O.loose_trie(same)["num_nodes"][0] == m
    distinct = np.arange(5 * m).reshape(5, m)
    assert O.loose_trie(distinct)["num_nodes"][0] == 5 * m
    one = O.loose_trie(np.array([[4, 4, 4]]))
    assert one["parent"][0].tolist() == [-1, 0, 1]
    with pytest.raises(ValueError):
        O.loose_trie(np.array([[1, -1]]))


# --------------------------------------------------------------------------
# a6: soft gate
# --------------------------------------------------------------------------

def _gate_from_golden(g, case):
    tr = g["tree"]
    root = np.array([g["root_logits"]], dtype=np.float32)
    nodes = np.array([g["node_logits"]], dtype=np.float32)
    hid_root = np.zeros((1, 2), dtype=np.float32)
    hid_nodes = np.arange(10, dtype=np.float32).reshape(1, 5, 2)
    return O.soft_gate(np.array([tr["tokens"]]), np.array([tr["parent"]]),
                       np.array([tr["num_nodes"]]), np.array([tr["gamma"]]),
                       root, nodes, hid_root, hid_nodes,
                       gamma_thr=case["gamma"], kappa=case["kappa"],
                       window=case["window"], return_masks=True)


def test_gate_golden():
    g = json.load(open(os.path.join(GOLDEN, "gate_small.json")))
    tr = O.loose_trie(np.array(g["spans"]))
    assert tr["tokens"][0].tolist()[:5] == g["tree"]["tokens"]
    assert tr["gamma"][0].tolist() == g["tree"]["gamma"]
    ne = g["normalized_entropy"]
    ent = O.sense_oracle._softmax_entropy(np.array([g["root_logits"], [0, 0, 0, 0], [9, 0, 0, 0]],
                                                   dtype=np.float64)) / math.log(4)
    np.testing.assert_allclose(ent, [ne["root"], ne["uniform"], ne["peak9"]], rtol=1e-4)
    for case in g["cases"]:
        out = _gate_from_golden(g, case)
        for key in ("B_em", "B_ent", "B_topk", "B_con", "G"):
            if key in case:
                assert out[key][0].tolist() == case[key], key
        assert out["i_star"][0] == case["i_star"]
        assert out["L_star"][0] == case["L_star"]
        assert out["n_accept"][0] == case["L_star"] + 1
        assert out["accepted"][0][:case["L_star"] + 1].tolist() == case["accepted"]
        assert out["next_node"][0] == case["next_node"]
        assert out["next_anchor"][0] == case["next_anchor"]
        assert out["h_next"][0].tolist() == [2.0 * case["next_node"], 2.0 * case["next_node"] + 1]


def test_entropy_closed_forms():
    v = 1000
    ent = O.sense_oracle._softmax_entropy(np.zeros((1, v)))
    assert abs(ent[0] / math.log(v) - 1.0) < 1e-12
    for n1, a, b in [(1, 7.0, 0.0), (5, 2.0, -1.0), (300, 0.5, 0.0)]:
        x = np.full(v, b)
        x[:n1] = a
        z = n1 * math.exp(a) + (v - n1) * math.exp(b)
        pa, pb = math.exp(a) / z, math.exp(b) / z
        closed = -(n1 * pa * math.log(pa) + (v - n1) * pb * math.log(pb))
        assert abs(O.sense_oracle._softmax_entropy(x[None])[0] - closed) < 1e-12
    scipy_stats = pytest.importorskip("scipy.stats")
    x = np.random.default_rng(0).standard_normal((4, 333)) * 3
    p = np.exp(x - x.max(1, keepdims=True))
    p /= p.sum(1, keepdims=True)
    np.testing.assert_allclose(O.sense_oracle._softmax_entropy(x), scipy_stats.entropy(p, axis=1),
                               rtol=1e-12)


def test_topk_membership_vs_torch():
    x = np.random.default_rng(1).standard_normal((50, 300)).astype(np.float32)
    tok = np.random.default_rng(2).integers(0, 300, size=50)
    for kappa in (1, 3, 10):
        ref = torch.topk(torch.from_numpy(x), kappa, dim=1).indices.numpy()
        want = np.array([tok[i] in ref[i] for i in range(50)])
        assert (O.sense_oracle._in_topk(x, tok, kappa) == want).all()


def _planted_case(seed, k=6, m=5, v=16):
    rng = np.random.default_rng(seed)
    spans = _rand_spans(rng, k, m, 4)
    tr = O.loose_trie(spans[None])
    cap = k * m
    root = synth.gate_logits(1, 1, v, seed=seed)[:, 0].clone()
    nodes = synth.gate_logits(1, cap, v, seed=seed + 1)
    synth.plant_gate_rows(root, nodes, torch.from_numpy(tr["tokens"]),
                          torch.from_numpy(tr["parent"]), torch.from_numpy(tr["num_nodes"]),
                          seed=seed)
    hid_r = np.zeros((1, 3), np.float32)
    hid_n = np.random.default_rng(seed).standard_normal((1, cap, 3)).astype(np.float32)
    return spans, tr, root.numpy(), nodes.numpy(), hid_r, hid_n


@pytest.mark.parametrize("seed", range(6))
def test_gate_greedy_special_case(seed):
    """gamma >= 1 disables the rescue: G = B_em, the exact-match rule."""
    spans, tr, root, nodes, hr, hn = _planted_case(seed)
    out = O.soft_gate(tr["tokens"], tr["parent"], tr["num_nodes"], tr["gamma"], root, nodes,
                      hr, hn, gamma_thr=1.0, return_masks=True)
    k, m = spans.shape
    best_len, best_i = -1, 0
    for i in range(k):
        n_ok = 0
        row = root[0]
        for j in range(m):
            if int(np.argmax(row)) != spans[i, j]:
                break
            n_ok += 1
            row = nodes[0, tr["gamma"][0][i, j]]
        assert out["G"][0][i].tolist() == out["B_em"][0][i].tolist()
        if n_ok - 1 > best_len:
            best_len, best_i = n_ok - 1, i
    assert out["L_star"][0] == best_len and out["i_star"][0] == best_i


@pytest.mark.parametrize("seed", range(3))
def test_gate_accept_all_special_case(seed):
    spans, tr, root, nodes, hr, hn = _planted_case(seed)
    out = O.soft_gate(tr["tokens"], tr["parent"], tr["num_nodes"], tr["gamma"], root, nodes,
                      hr, hn, gamma_thr=-1.0, kappa=root.shape[-1])
    assert (out["G"] == 1).all()
    assert out["L_star"][0] == spans.shape[1] - 1 and out["i_star"][0] == 0


@pytest.mark.parametrize("w", [1, 3, 6])
def test_gate_con_matches_torch_conv1d(w):
    spans, tr, root, nodes, hr, hn = _planted_case(7)
    out = O.soft_gate(tr["tokens"], tr["parent"], tr["num_nodes"], tr["gamma"], root, nodes,
                      hr, hn, window=w, return_masks=True)
    m = spans.shape[1]
    bbar = torch.nn.functional.pad(1.0 - torch.from_numpy(out["B_em"][0]).double(), (0, w), value=1.0)
    r = torch.nn.functional.conv1d(bbar[:, None], torch.ones(1, 1, w, dtype=torch.float64))[:, 0]
    want = (r[:, 1:m + 1] == 0).numpy().astype(np.uint8)
    assert out["B_con"][0].tolist() == want.tolist()


def test_gate_cap_truncation():
    spans = np.array([[1, 2, 3, 4], [5, 6, 7, 8]])
    tr = O.loose_trie(spans, node_cap=5)  # keeps 1,2,3,4 and 5
    v = 10
    root = np.zeros((1, v), np.float32)
    root[0, 1] = 50.0
    nodes = np.zeros((1, 5, v), np.float32)
    for n, t in enumerate([2, 3, 4]):
        nodes[0, n, t] = 50.0
    out = O.soft_gate(tr["tokens"], tr["parent"], tr["num_nodes"], tr["gamma"], root, nodes,
                      np.zeros((1, 1)), np.zeros((1, 5, 1)), gamma_thr=-1.0, kappa=v)
    assert out["G"][0].tolist() == [[1, 1, 1, 1], [1, 0, 0, 0]]
    assert out["i_star"][0] == 0 and out["L_star"][0] == 3


# --------------------------------------------------------------------------
# tree attention mask over a static KV cache (App. C.6 Eq. 20)
# --------------------------------------------------------------------------

def test_tree_mask_full_chain_is_shifted_causal():
    # one span -> a chain: every draft token sees the committed tokens and
    # the draft tokens up to itself, i.e. the textbook causal mask
    m, cache, depth = 5, 16, 7
    tr = O.loose_trie(np.array([[3, 1, 4, 1, 5, 9, 2]]), mask_bits=True)
    M = O.mask_from_bits(tr["mask_bits"][0], tr["num_nodes"][0])
    np.testing.assert_array_equal(M, np.tril(np.ones((depth, depth), dtype=np.int64)))
    full = O.tree_mask_full(M, m, cache)
    causal = np.triu(np.full((m + depth, m + depth), -np.inf), k=1)[m:]
    want = np.full((depth, cache), -np.inf)
    want[:, :m + depth] = causal
    np.testing.assert_array_equal(full, want)


def test_tree_mask_full_golden():
    g = json.load(open(os.path.join(GOLDEN, "trie_small.json")))
    u = g["uncapped"]
    words = np.array(u["mask_words"], dtype=np.uint32)[:, None]
    M = O.mask_from_bits(words, u["num_nodes"])
    _, _, mask_alg3, _ = O.loose_trie_alg3(np.array(g["spans"]))
    np.testing.assert_array_equal(M, mask_alg3)
    full = O.tree_mask_full(M, 2, 14, rows=12)
    # node 5 is the path (5, 4, 0) = nodes 0, 4, 5: committed columns 0, 1
    # plus cache positions 2 + {0, 4, 5}
    assert np.nonzero(full[5] == 0)[0].tolist() == [0, 1, 2, 6, 7]
    # every row sees m + depth + 1 columns; padding rows see the m committed
    assert (full[:9] == 0).sum(axis=1).tolist() == [2 + d + 1 for d in u["depth"]]
    assert (full[9:] == 0).sum(axis=1).tolist() == [2, 2, 2]
    assert np.all(full[9:, :2] == 0)
    with pytest.raises(ValueError):
        O.tree_mask_full(M, 6, 14)


@pytest.mark.parametrize("seed", range(3))
def test_tree_mask_full_attention_equals_per_path_causal(seed):
    # Tree attention with M_full over the cache gives each draft token the
    # same output as causal attention over its own sequence (committed
    # tokens, then its root path), computed here by torch's reference SDPA.
    rng = np.random.default_rng(300 + seed)
    spans = _rand_spans(rng, 6, 4, 3)
    tr = O.loose_trie(spans, mask_bits=True)
    L = int(tr["num_nodes"][0])
    M = O.mask_from_bits(tr["mask_bits"][0], L)
    m, cache, hd = 5, 5 + L + 3, 8
    g = torch.Generator().manual_seed(seed)
    q = torch.randn(L, hd, generator=g, dtype=torch.float64)
    kc = torch.randn(cache, hd, generator=g, dtype=torch.float64)
    vc = torch.randn(cache, hd, generator=g, dtype=torch.float64)
    full = torch.from_numpy(O.tree_mask_full(M, m, cache))
    tree_out = torch.softmax(q @ kc.T / math.sqrt(hd) + full, dim=-1) @ vc
    par = tr["parent"][0]
    for i in range(L):
        path, p = [], i
        while p >= 0:
            path.append(p)
            p = par[p]
        cols = list(range(m)) + [m + n for n in reversed(path)]
        qs = torch.zeros(len(cols), hd, dtype=torch.float64)
        qs[-1] = q[i]
        ref = torch.nn.functional.scaled_dot_product_attention(
            qs[None], kc[cols][None], vc[cols][None], is_causal=True)[0, -1]
        torch.testing.assert_close(tree_out[i], ref, rtol=1e-12, atol=1e-12)


def _bf(x):
    return _bits(torch.from_numpy(np.asarray(x, np.float32)).to(torch.bfloat16))


def test_tree_attention_matches_sdpa_with_float_mask():
    rng = np.random.default_rng(31)
    spans = _rand_spans(rng, 8, 5, 3)
    tr = O.loose_trie(spans, mask_bits=True)
    L = int(tr["num_nodes"][0])
    M = O.mask_from_bits(tr["mask_bits"][0], L)
    H, D, m = 3, 16, 7
    q = _bf(rng.standard_normal((H, L, D)))
    k = _bf(rng.standard_normal((H, m + L + 5, D)))
    v = _bf(rng.standard_normal((H, m + L + 5, D)))
    got = O.tree_attention(q, k, v, m, M, 0.25)
    qt, kt, vt = (torch.from_numpy(O.bf16_bits_to_f64(a)) for a in (q, k, v))
    full = torch.from_numpy(O.tree_mask_full(M, m, m + L))
    ref = torch.nn.functional.scaled_dot_product_attention(
        qt, kt[:, :m + L], vt[:, :m + L], attn_mask=full, scale=0.25)
    np.testing.assert_allclose(got, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_tree_attention_chain_is_causal_attention():
    rng = np.random.default_rng(32)
    L, m, H, D = 6, 4, 2, 8
    M = np.tril(np.ones((L, L), dtype=np.int64))
    q = _bf(rng.standard_normal((H, L, D)))
    k = _bf(rng.standard_normal((H, m + L, D)))
    v = _bf(rng.standard_normal((H, m + L, D)))
    got = O.tree_attention(q, k, v, m, M, 1 / np.sqrt(D))
    qt, kt, vt = (torch.from_numpy(O.bf16_bits_to_f64(a)) for a in (q, k, v))
    # causal attention over the whole sequence; the last L rows are the tree
    qfull = torch.cat([torch.zeros(H, m, D, dtype=torch.float64), qt], dim=1)
    ref = torch.nn.functional.scaled_dot_product_attention(qfull, kt, vt, is_causal=True)[:, m:]
    np.testing.assert_allclose(got, ref.numpy(), rtol=1e-12, atol=1e-12)
