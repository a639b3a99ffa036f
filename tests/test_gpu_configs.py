"""Parity at the workloads' full sizes, in the launch configuration bench.py
times (one call per query batch, the same k, m, cap and gate parameters).

Retrieval is checked exhaustively for a seeded subset of queries: the oracle
scores every key of the store (copied to the host in 65,536-row slices) and
the full top-k rule applies (4 steps of the 1M-key store, 1 step of the
137 GB store, every query of one 16-query batch of the 4M-key store and of
the 64-query batches of the 2M-key sweeps, every query of the tiny store).  The other checked queries use sampled outputs the
oracle computes one by one: (a) every key returned, (b) every key of the
query's source cluster and (c) a seeded random sample of the store (about
1 GB of keys).  Their returned scores must match, the order must agree, no
sampled key may beat the returned k-th by more than the tolerance, and the
query's source key must be returned.  Gather, tree and gate run on seeded
inputs drawn from each workload's distributions and are compared bit for bit
(gate: seeded query subsets at the full vocabulary).
"""
import gc

import numpy as np
import pytest
import torch

import oracle as O
import synth
from synth.workloads import WORKLOADS
from tests.parity import SCORE_TOL, bits, check_topk, host

pytestmark = pytest.mark.gpu
cuda = pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")
GATE = dict(gamma=0.05, topk=3, window=6, tau=0)


@pytest.fixture(scope="module")
def S():
    import paper_2606_00021_gb300 as S
    S.lib()
    return S


def _free():
    gc.collect()
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def _spans(cfg, n, seed, dev):
    if cfg["zipf"]:
        return synth.spans_zipf(n, cfg["m"], cfg["vocab"], 1.1, seed=seed, device=dev)
    return synth.spans_uniform(n, cfg["m"], cfg["vocab"], seed=seed, device=dev)


def _check_query(keys, assign_h, q_bits, src, sc, ix, k, sample_rows):
    """Sampled parity of one query's top-k (see the module docstring)."""
    dev = keys.device
    ret = host(ix).astype(np.int64)
    assert len(set(ret.tolist())) == k and ret.min() >= 0 and ret.max() < keys.shape[0]
    cluster = np.nonzero(assign_h == assign_h[src])[0]
    cand = np.unique(np.concatenate([ret, cluster, sample_rows]))
    sub = keys.index_select(0, torch.from_numpy(cand).to(dev))
    s = O.scores(bits(sub), q_bits)[0]
    pos = {int(r): i for i, r in enumerate(cand)}
    s_ret = np.array([s[pos[int(r)]] for r in ret])
    err = np.abs(host(sc).astype(np.float64) - s_ret)
    assert err.max() <= SCORE_TOL, f"score error {err.max():.3g}"
    assert np.all(np.diff(s_ret) <= SCORE_TOL), "order disagrees beyond tolerance"
    kth = s_ret.min()
    others = np.setdiff1d(cand, ret)
    missed = s[[pos[int(r)] for r in others]] if others.size else np.zeros(0)
    assert missed.size == 0 or missed.max() <= kth + SCORE_TOL, \
        f"a key scoring {missed.max():.6f} beats the returned k-th {kth:.6f}"
    assert src in set(ret.tolist()), "the query's source key was not returned"


def _exhaustive_scores(keys, q_bits):
    """The oracle's scores of every key of the store for the given queries
    (fp64 [q, n]), the keys copied to the host one 65,536-row slice at a
    time."""
    n = keys.shape[0]
    out = np.empty((q_bits.shape[0], n), dtype=np.float64)
    for lo in range(0, n, 65536):
        hi = min(n, lo + 65536)
        out[:, lo:hi] = O.scores(bits(keys[lo:hi]), q_bits)
    return out


# queries checked against every key of the store: (query batches, queries per batch)
EXHAUSTIVE = {"tiny_4k": (1, 8), "llama7b_1m": (4, 1), "llama70b_8m": (1, 1),
              "qwen7b_4m": (1, 16), "sweep_2m_k16": (1, 64), "sweep_2m_k64": (1, 64),
              "sweep_2m_k256": (1, 64)}


@cuda
@pytest.mark.parametrize("name", ["tiny_4k", "llama7b_1m", "qwen7b_4m", "llama70b_8m",
                                  "sweep_2m_k16", "sweep_2m_k64", "sweep_2m_k256"])
def test_full_size_retrieval(S, name):
    cfg = WORKLOADS[name]
    dev = torch.device("cuda")
    n, d, q, k = cfg["n"], cfg["d"], cfg["q"], cfg["k"]
    keys, assign = synth.clustered_unit_keys(n, d, cfg["clusters"], seed=0, device=dev,
                                             return_assign=True)
    spans = _spans(cfg, n, 0, dev)
    # single-query workloads: a seeded subset of steps (16; 4 for the 137 GB store)
    batches = (4 if n * d > (1 << 35) else 16) if q == 1 else 1
    qs, src = synth.noisy_queries(keys, q * batches, noise=0.05, seed=1)
    ds = S.sense_datastore_build(keys, spans)
    ws = S.alloc_workspace(S.sense_retrieve_workspace_bytes(ds, q, k))
    assign_h = host(assign)
    rng = np.random.default_rng(7)
    n_sample = min(n, (1 << 30) // (d * 2))
    sample_rows = np.sort(rng.choice(n, size=n_sample, replace=False))
    results = []
    for b in range(batches):
        qb = qs[b * q:(b + 1) * q].contiguous()
        sc, ix = S.sense_retrieve_topk(ds, qb, k, workspace=ws)
        torch.cuda.synchronize()
        assert S.sense_device_status(clear=True) == 0
        results.append((qb, host(sc), host(ix)))
    ex_b, ex_q = EXHAUSTIVE.get(name, (0, 0))
    checked = exhaustive = 0
    if ex_b:
        q_bits = np.concatenate([bits(results[b][0][:ex_q]) for b in range(ex_b)])
        full = _exhaustive_scores(keys, q_bits)
        row = 0
        for b in range(ex_b):
            _, sc_h, ix_h = results[b]
            for qi in range(ex_q):
                check_topk(sc_h[qi], ix_h[qi], full[row], k)
                assert int(src[b * q + qi]) in set(ix_h[qi].tolist())
                row += 1
                exhaustive += 1
        del full
    for b in range(batches):
        qb, sc_h, ix_h = results[b]
        # every query of the batch (up to 64) not already checked exhaustively
        pick = range(q) if q <= 64 else sorted(rng.choice(q, size=64, replace=False).tolist())
        for qi in pick:
            if b < ex_b and qi < ex_q:
                continue
            _check_query(keys, assign_h, bits(qb[qi:qi + 1]), int(src[b * q + qi]),
                         torch.from_numpy(sc_h[qi]), torch.from_numpy(ix_h[qi]), k, sample_rows)
            checked += 1
    assert checked + exhaustive >= 3
    assert exhaustive == ex_b * ex_q
    del ds, keys, spans, assign, qs, ws
    _free()


@cuda
@pytest.mark.parametrize("name", ["tiny_4k", "llama7b_1m", "qwen7b_4m", "llama70b_8m",
                                  "sweep_2m_k16", "sweep_2m_k64", "sweep_2m_k256"])
def test_full_size_gather_and_tree(S, name):
    cfg = WORKLOADS[name]
    dev = torch.device("cuda")
    n, q, k, m = cfg["n"], cfg["q"], cfg["k"], cfg["m"]
    # the datastore's key matrix does not matter here: one shared row of keys
    keys = torch.zeros(n, 8, dtype=torch.bfloat16, device=dev)
    spans = _spans(cfg, n, 3, dev)
    ds = S.sense_datastore_build(keys, spans)
    g = torch.Generator(device=dev).manual_seed(11)
    idx = torch.randint(0, n, (q, k), generator=g, device=dev, dtype=torch.int32)
    drafts = S.sense_gather_drafts(ds, idx)
    tree = S.sense_build_tree(drafts, node_cap=cfg["cap"])
    torch.cuda.synchronize()
    assert S.sense_device_status(clear=True) == 0
    sp_h = host(spans)
    want_d = O.gather_drafts(sp_h, host(idx))
    np.testing.assert_array_equal(host(drafts), want_d)
    sub = range(q) if q <= 64 else range(0, q, max(1, q // 64))
    for qi in sub:
        want = O.loose_trie(want_d[qi:qi + 1], node_cap=cfg["cap"])
        for key in ("num_nodes", "tokens", "parent", "depth", "gamma"):
            np.testing.assert_array_equal(host(tree[key][qi:qi + 1]), want[key], err_msg=key)
    del ds, keys, spans
    _free()


@cuda
@pytest.mark.parametrize("name,nq,plant,seed", [
    ("tiny_4k", 8, True, 7), ("llama7b_1m", 4, False, 5), ("llama7b_1m", 4, True, 5),
    ("qwen7b_4m", 3, True, 7), ("llama70b_8m", 3, True, 7), ("sweep_2m_k16", 4, True, 7),
    ("sweep_2m_k64", 2, True, 7), ("sweep_2m_k256", 1, True, 5), ("sweep_2m_k256", 1, False, 5),
])
def test_full_size_gate(S, name, nq, plant, seed):
    """Gate at the workload's vocabulary, hidden size, k, m and cap on seeded
    trees (spans drawn from a small vocabulary so that prefixes are shared).
    The logits seeds are chosen so that no query has a normalised entropy
    within the 1e-4 band of the threshold (the fixture check below allows at
    most one such query per case, and never all of them)."""
    cfg = WORKLOADS[name]
    dev = torch.device("cuda")
    k, m, v, d = cfg["k"], cfg["m"], cfg["vocab"], cfg["d"]
    rng = np.random.default_rng(k * 7 + m)
    base = rng.integers(0, 8, size=(nq, max(1, k // 4), m))
    sp = np.empty((nq, k, m), dtype=np.int32)
    for qi in range(nq):
        rows = base[qi][rng.integers(0, base.shape[1], size=k)].copy()
        for r in range(k):
            cut = int(rng.integers(0, m + 1))
            rows[r, cut:] = rng.integers(0, 8, size=m - cut)
        sp[qi] = rows
    tr = O.loose_trie(sp, node_cap=cfg["cap"])
    cap = tr["tokens"].shape[1]
    root = synth.gate_logits(nq, 1, v, seed=seed)[:, 0].contiguous()
    nodes = synth.gate_logits(nq, cap, v, seed=seed + 1)
    if plant:
        synth.plant_gate_rows(root, nodes, torch.from_numpy(tr["tokens"]),
                              torch.from_numpy(tr["parent"]), torch.from_numpy(tr["num_nodes"]),
                              seed=seed)
    hr = synth.gate_hidden(nq, 1, d, seed=5)[:, 0].contiguous()
    hn = synth.gate_hidden(nq, cap, d, seed=6)
    tree = {key: torch.from_numpy(tr[key]).to(dev) for key in
            ("num_nodes", "tokens", "parent", "gamma")}
    got = S.sense_soft_gate(tree, root.to(dev), nodes.to(dev), hr.to(dev), hn.to(dev),
                            want_G=True, **GATE)
    torch.cuda.synchronize()
    want = O.soft_gate(tr["tokens"], tr["parent"], tr["num_nodes"], tr["gamma"], host(root),
                       host(nodes), bits(hr), bits(hn), gamma_thr=GATE["gamma"],
                       kappa=GATE["topk"], window=GATE["window"], tau=GATE["tau"],
                       ent_band=1e-4)
    ok = ~want["ambiguous"]
    assert ok.any() and (~ok).sum() <= 1, "fixture: too many near-threshold entropies"
    for key in ("i_star", "L_star", "n_accept", "next_node", "next_anchor"):
        np.testing.assert_array_equal(host(got[key])[ok], want[key][ok], err_msg=key)
    np.testing.assert_array_equal(host(got["accepted"])[ok], want["accepted"][ok])
    np.testing.assert_array_equal(host(got["G"])[ok], want["G"][ok])
    np.testing.assert_array_equal(bits(got["h_next"])[ok], want["h_next"][ok])
    del got, nodes, hn
    _free()
