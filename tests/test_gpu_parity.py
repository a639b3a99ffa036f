"""GPU-vs-oracle parity of every step of the path, through the C ABI.

Sizes are small enough for the oracle to finish in seconds but span several
tiles, the sampled-threshold path and ragged tails.  Inputs come from the
seeded generators in ``synth``; expected values only from ``oracle``.
"""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from tests.parity import SCORE_TOL, bits, check_topk, host

pytestmark = pytest.mark.gpu

cuda = pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")


@pytest.fixture(scope="module")
def S():
    import paper_2606_00021_gb300 as S
    S.lib()
    return S


def _clear(S):
    return S.sense_device_status(clear=True)


# ---------------------------------------------------------------- retrieval

@cuda
@pytest.mark.parametrize("n,d,q,k,clusters", [
    (4096, 4096, 8, 8, 64),      # tiny: all keys in one pass
    (5000, 512, 3, 17, 16),      # ragged last tile, no sampling
    (131072 + 77, 512, 1, 32, 256),   # sampled threshold path, ragged
    (200003, 256, 5, 64, 512),   # sampled, several queries
    (70000, 1024, 2, 1, 64),     # k = 1
])
def test_retrieve_matches_oracle(S, n, d, q, k, clusters):
    dev = torch.device("cuda")
    keys = synth.clustered_unit_keys(n, d, clusters, seed=n % 97, device=dev)
    spans = synth.spans_uniform(n, 8, 32000, seed=1, device=dev)
    qs, _ = synth.noisy_queries(keys, q, seed=n % 13)
    ds = S.sense_datastore_build(keys, spans)
    sc, ix = S.sense_retrieve_topk(ds, qs, k)
    torch.cuda.synchronize()
    assert _clear(S) == 0
    full = O.scores(bits(keys), bits(qs))
    for qi in range(q):
        check_topk(host(sc[qi]), host(ix[qi]), full[qi], k)


@cuda
@pytest.mark.parametrize("n,d,q,k,clusters", [
    (4096, 4096, 16, 8, 64),        # tensor path, one pass, no sampling
    (5000, 512, 9, 17, 16),         # q padded 9 -> 16, ragged tile
    (131072 + 77, 512, 33, 32, 256),  # sampled, nq = 48
    (200003, 256, 64, 64, 512),     # sampled, q = 64
    (70000, 1024, 128, 5, 64),      # full 128-query group
    (66000, 320, 130, 16, 64),      # two groups (128 + 2), d not a multiple of 64
])
def test_retrieve_tensor_path_matches_oracle(S, n, d, q, k, clusters):
    dev = torch.device("cuda")
    keys = synth.clustered_unit_keys(n, d, clusters, seed=n % 89, device=dev)
    spans = synth.spans_uniform(n, 4, 32000, seed=1, device=dev)
    qs, _ = synth.noisy_queries(keys, q, seed=n % 11)
    ds = S.sense_datastore_build(keys, spans)
    sc, ix = S.sense_retrieve_topk(ds, qs, k)
    torch.cuda.synchronize()
    assert _clear(S) == 0
    full = O.scores(bits(keys), bits(qs))
    for qi in range(q):
        check_topk(host(sc[qi]), host(ix[qi]), full[qi], k)


@cuda
@pytest.mark.parametrize("n,d,q,k", [(20000, 256, 1, 64), (20000, 256, 8, 17),
                                     (150000, 128, 3, 100), (4096, 64, 2, 4096 // 4),
                                     (20000, 256, 16, 64), (150000, 192, 40, 100),
                                     (9000, 64, 129, 33), (30000, 192, 24, 50)])
def test_retrieve_lattice_bit_exact(S, n, d, q, k):
    """Lattice entries make every fp32 sum exact: scores, order and ties
    (lower index first) must equal the oracle bit for bit."""
    dev = torch.device("cuda")
    keys = synth.lattice_rows(n, d, seed=3, device=dev)
    qs = synth.lattice_rows(q, d, seed=4, device=dev)
    spans = synth.spans_uniform(n, 4, 100, seed=1, device=dev)
    ds = S.sense_datastore_build(keys, spans)
    sc, ix = S.sense_retrieve_topk(ds, qs, k)
    torch.cuda.synchronize()
    assert _clear(S) == 0
    ov, oi = O.topk(O.scores(bits(keys), bits(qs)), k)
    np.testing.assert_array_equal(host(ix), oi)
    np.testing.assert_array_equal(host(sc).astype(np.float64), ov)


@cuda
def test_retrieve_k_equals_n_and_repeat(S):
    dev = torch.device("cuda")
    n, d = 300, 128
    keys = synth.clustered_unit_keys(n, d, 4, seed=2, device=dev)
    spans = synth.spans_uniform(n, 2, 50, seed=2, device=dev)
    qs, _ = synth.noisy_queries(keys, 2, seed=2)
    ds = S.sense_datastore_build(keys, spans)
    ws = S.alloc_workspace(S.sense_retrieve_workspace_bytes(ds, 2, n))
    a = S.sense_retrieve_topk(ds, qs, n, workspace=ws)
    b = S.sense_retrieve_topk(ds, qs, n, workspace=ws)  # workspace reuse
    torch.cuda.synchronize()
    assert torch.equal(a[1], b[1]) and torch.equal(a[0], b[0])
    full = O.scores(bits(keys), bits(qs))
    for qi in range(2):
        assert sorted(host(a[1][qi]).tolist()) == list(range(n))
        check_topk(host(a[0][qi]), host(a[1][qi]), full[qi], n)


@cuda
def test_datastore_normalize(S):
    dev = torch.device("cuda")
    x = synth.gaussian_rows_f32(1000, 512, seed=5, device=dev) * 3.0
    x[7] = 0.0
    spans = synth.spans_uniform(1000, 4, 10, seed=5, device=dev)
    ds = S.sense_datastore_build(x, spans, normalize=True)
    got = bits(S.sense_datastore_keys(ds))
    torch.cuda.synchronize()
    want = O.normalize_keys_bf16(host(x))
    diff = np.abs(got.astype(np.int32) - want.astype(np.int32))
    assert diff.max() <= 1 and (diff == 0).mean() > 0.9999
    assert (got[7] == 0).all()


# ---------------------------------------------------------------- gather

@cuda
def test_gather_plain_and_bad_index(S):
    dev = torch.device("cuda")
    n, m = 1000, 16
    keys = synth.clustered_unit_keys(n, 64, 4, seed=1, device=dev)
    spans = synth.spans_zipf(n, m, 32000, seed=1, device=dev)
    ds = S.sense_datastore_build(keys, spans)
    g = torch.Generator().manual_seed(0)
    idx = torch.randint(0, n, (5, 32), generator=g, dtype=torch.int32)
    idx[2, 5] = -1
    idx[4, 31] = n
    _clear(S)
    out = S.sense_gather_drafts(ds, idx.to(dev))
    st = S.sense_device_status(clear=True)
    assert st & S.DEVST_BAD_INDEX
    want = O.gather_drafts(host(spans), host(idx))
    np.testing.assert_array_equal(host(out), want)


@cuda
@pytest.mark.parametrize("k,keep,force", [(32, 32, False), (32, 10, True), (7, 3, False),
                                          (256, 100, True), (1, 1, True)])
def test_gather_anchor_rerank(S, k, keep, force):
    dev = torch.device("cuda")
    n, m = 2000, 8
    keys = synth.clustered_unit_keys(n, 64, 4, seed=1, device=dev)
    spans = synth.spans_uniform(n, m, 6, seed=3, device=dev)  # tiny vocab: many matches
    ds = S.sense_datastore_build(keys, spans)
    g = torch.Generator().manual_seed(k)
    q = 6
    idx = torch.stack([torch.randperm(n, generator=g)[:k] for _ in range(q)]).to(torch.int32)
    anchor = torch.randint(0, 6, (q,), generator=g, dtype=torch.int32)
    out = S.sense_gather_drafts(ds, idx.to(dev), anchor=anchor.to(dev), n_keep=keep,
                                force_anchor=force)
    torch.cuda.synchronize()
    want = O.gather_drafts(host(spans), host(idx), anchor=host(anchor), n_keep=keep,
                           force_anchor=force)
    np.testing.assert_array_equal(host(out), want)


# ---------------------------------------------------------------- tree

def _tree_spans(q, k, m, vocab, seed):
    rng = np.random.default_rng(seed)
    out = np.empty((q, k, m), dtype=np.int32)
    for qi in range(q):
        base = rng.integers(0, vocab, size=(max(1, k // 4), m))
        rows = base[rng.integers(0, base.shape[0], size=k)].copy()
        for r in range(k):
            cut = int(rng.integers(0, m + 1))
            rows[r, cut:] = rng.integers(0, vocab, size=m - cut)
        out[qi] = rows
    return out


def _check_tree(got, want, q, cap):
    for key in ("num_nodes", "tokens", "parent", "depth", "gamma"):
        np.testing.assert_array_equal(host(got[key]), want[key], err_msg=key)
    if "mask_bits" in want:
        np.testing.assert_array_equal(host(got["mask_bits"]).view(np.uint32), want["mask_bits"])


@cuda
@pytest.mark.parametrize("q,k,m,vocab,cap", [
    (3, 8, 8, 5, 0), (4, 32, 16, 3, 64), (2, 256, 16, 4, 0), (2, 256, 16, 50, 128),
    (3, 1, 5, 3, 0), (2, 64, 1, 10, 0), (2, 1024, 8, 3, 0), (2, 300, 27, 2, 4000),
    (2, 512, 16, 3, 7), (1, 17, 32, 2, 1),
    (2, 128, 32, 3, 200), (1, 128, 8, 2, 0), (2, 129, 4, 3, 50),  # small-path boundary
])
def test_tree_matches_oracle(S, q, k, m, vocab, cap):
    dev = torch.device("cuda")
    sp = _tree_spans(q, k, m, vocab, seed=q * 1000 + k + m)
    mask = (k * m <= 1024)
    got = S.sense_build_tree(torch.from_numpy(sp).to(dev), node_cap=cap, mask_bits=mask)
    torch.cuda.synchronize()
    assert _clear(S) == 0
    want = O.loose_trie(sp, node_cap=cap, mask_bits=mask)
    _check_tree(got, want, q, cap)


@cuda
def test_tree_special_cases_and_bad_token(S):
    dev = torch.device("cuda")
    m = 6
    same = np.tile(np.arange(m, dtype=np.int32), (1, 9, 1))
    got = S.sense_build_tree(torch.from_numpy(same).to(dev))
    torch.cuda.synchronize()
    assert int(got["num_nodes"][0]) == m
    sp = _tree_spans(2, 4, 4, 3, seed=1)
    sp[1, 2, 3] = -5
    _clear(S)
    got = S.sense_build_tree(torch.from_numpy(sp).to(dev))
    st = S.sense_device_status(clear=True)
    assert st & S.DEVST_BAD_TOKEN
    want0 = O.loose_trie(sp[:1])
    assert int(got["num_nodes"][1]) == 0 and (host(got["gamma"][1]) == -1).all()
    np.testing.assert_array_equal(host(got["tokens"][0]), want0["tokens"][0])


# ---------------------------------------------------------------- tree mask (Eq. 20)

def _mask_want(sp, cap, prefix, cache_len):
    tr = O.loose_trie(sp, node_cap=cap, mask_bits=True)
    rows = tr["tokens"].shape[1]
    out = np.empty((sp.shape[0], rows, cache_len))
    for qi in range(sp.shape[0]):
        nn = int(tr["num_nodes"][qi])
        M = O.mask_from_bits(tr["mask_bits"][qi], nn)
        out[qi] = O.tree_mask_full(M, int(prefix[qi]), cache_len, rows=rows)
    return out


@cuda
@pytest.mark.parametrize("q,k,m,vocab,cap,cache_len", [
    (3, 8, 8, 5, 64, 256), (2, 32, 16, 3, 128, 1027), (2, 64, 8, 4, 0, 600),
    (1, 1, 5, 3, 0, 5), (4, 16, 4, 2, 33, 97),
])
def test_tree_mask_full_matches_oracle(S, q, k, m, vocab, cap, cache_len):
    dev = torch.device("cuda")
    sp = _tree_spans(q, k, m, vocab, seed=q * 31 + k + cache_len)
    tree = S.sense_build_tree(torch.from_numpy(sp).to(dev), node_cap=cap, mask_bits=True)
    nn = host(tree["num_nodes"])
    rng = np.random.default_rng(cache_len)
    # committed lengths from 0 up to the largest that fits (m + L == cache_len)
    prefix = np.array([int(rng.integers(0, cache_len - nn[qi] + 1)) for qi in range(q)],
                      dtype=np.int32)
    prefix[0] = cache_len - nn[0]
    if q > 1:
        prefix[1] = 0
    got = S.sense_tree_mask_full(tree, torch.from_numpy(prefix).to(dev), cache_len)
    torch.cuda.synchronize()
    assert _clear(S) == 0
    want = _mask_want(sp, cap, prefix, cache_len).astype(np.float32)
    np.testing.assert_array_equal(host(got), want)


@cuda
def test_tree_mask_full_flags_bad_length(S):
    dev = torch.device("cuda")
    sp = _tree_spans(3, 8, 6, 4, seed=5)
    tree = S.sense_build_tree(torch.from_numpy(sp).to(dev), node_cap=40, mask_bits=True)
    nn = host(tree["num_nodes"])
    cache_len = 64
    prefix = np.array([3, cache_len - nn[1] + 1, -1], dtype=np.int32)
    _clear(S)
    got = host(S.sense_tree_mask_full(tree, torch.from_numpy(prefix).to(dev), cache_len))
    st = S.sense_device_status(clear=True)
    assert st == S.DEVST_BAD_LENGTH
    assert np.all(got[1:] == -np.inf)
    want = _mask_want(sp[:1], 40, prefix[:1], cache_len).astype(np.float32)
    np.testing.assert_array_equal(got[:1], want)


# ---------------------------------------------------------------- gate

def _gate_case(q, k, m, v, d, cap, seed, plant=True):
    sp = _tree_spans(q, k, m, 6, seed=seed)
    tr = O.loose_trie(sp, node_cap=cap)
    capn = tr["tokens"].shape[1]
    root = synth.gate_logits(q, 1, v, seed=seed)[:, 0].contiguous()
    nodes = synth.gate_logits(q, capn, v, seed=seed + 1)
    if plant:
        synth.plant_gate_rows(root, nodes, torch.from_numpy(tr["tokens"]),
                              torch.from_numpy(tr["parent"]), torch.from_numpy(tr["num_nodes"]),
                              seed=seed)
    hr = synth.gate_hidden(q, 1, d, seed=seed)[:, 0].contiguous()
    hn = synth.gate_hidden(q, capn, d, seed=seed + 1)
    return sp, tr, root, nodes, hr, hn


@cuda
@pytest.mark.parametrize("q,k,m,v,cap,gamma,kappa,w,tau,unnorm", [
    (4, 8, 8, 1000, 0, 0.05, 3, 6, 0, False),
    (3, 16, 16, 4096, 64, 0.05, 3, 6, 0, False),
    (3, 5, 10, 2000, 0, 0.3, 10, 5, 1, False),
    (2, 32, 16, 32000, 64, 0.01, 2, 9, 0, False),
    (2, 8, 4, 512, 0, 1.5, 4, 2, 0, True),
    (2, 3, 16, 128, 0, -1.0, 16, 1, 0, False),
    (1, 32, 16, 32000, 64, 0.05, 3, 6, 0, False),   # one query: two blocks per row
    (1, 4, 4, 64, 0, 0.5, 16, 3, 1, False),         # slices of one float4, empty slices
    (1, 16, 8, 40000, 0, 0.05, 5, 4, 0, False),     # one block per row, three stages a warp
    (1, 16, 16, 128256, 64, 0.05, 3, 6, 0, False),  # one query, long rows: split rows merged
])
def test_gate_matches_oracle(S, q, k, m, v, cap, gamma, kappa, w, tau, unnorm):
    dev = torch.device("cuda")
    d = 64
    sp, tr, root, nodes, hr, hn = _gate_case(q, k, m, v, d, cap, seed=k * 31 + m + v)
    tree = {key: torch.from_numpy(tr[key]).to(dev) for key in
            ("num_nodes", "tokens", "parent", "gamma")}
    got = S.sense_soft_gate(tree, root.to(dev), nodes.to(dev), hr.to(dev), hn.to(dev),
                            gamma=gamma, topk=kappa, window=w, tau=tau,
                            unnormalized_entropy=unnorm, want_G=True)
    torch.cuda.synchronize()
    want = O.soft_gate(tr["tokens"], tr["parent"], tr["num_nodes"], tr["gamma"], host(root),
                       host(nodes), bits(hr), bits(hn), gamma_thr=gamma, kappa=kappa,
                       window=w, tau=tau, unnormalized_entropy=unnorm, ent_band=1e-4)
    ok = ~want["ambiguous"]
    assert ok.any() and (~ok).sum() <= 1, "fixture: too many near-threshold entropies"
    for key in ("i_star", "L_star", "n_accept", "next_node", "next_anchor"):
        np.testing.assert_array_equal(host(got[key])[ok], want[key][ok], err_msg=key)
    np.testing.assert_array_equal(host(got["accepted"])[ok], want["accepted"][ok])
    np.testing.assert_array_equal(host(got["G"])[ok], want["G"][ok])
    np.testing.assert_array_equal(bits(got["h_next"])[ok], want["h_next"][ok])


@cuda
def test_gate_golden_fixture(S):
    import json
    import os
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "gate_small.json")))
    dev = torch.device("cuda")
    tr = g["tree"]
    tree = {"tokens": torch.tensor([tr["tokens"]], dtype=torch.int32, device=dev),
            "parent": torch.tensor([tr["parent"]], dtype=torch.int32, device=dev),
            "num_nodes": torch.tensor([tr["num_nodes"]], dtype=torch.int32, device=dev),
            "gamma": torch.tensor([tr["gamma"]], dtype=torch.int32, device=dev)}
    root = torch.tensor([g["root_logits"]], dtype=torch.float32, device=dev)
    nodes = torch.tensor([g["node_logits"]], dtype=torch.float32, device=dev)
    hr = torch.zeros(1, 8, dtype=torch.bfloat16, device=dev)
    hn = torch.arange(40, dtype=torch.float32).reshape(1, 5, 8).to(torch.bfloat16).to(dev)
    for case in g["cases"]:
        got = S.sense_soft_gate(tree, root, nodes, hr, hn, gamma=case["gamma"],
                                topk=case["kappa"], window=case["window"], want_G=True)
        torch.cuda.synchronize()
        assert host(got["G"])[0].tolist() == case["G"]
        assert int(got["i_star"][0]) == case["i_star"]
        assert int(got["L_star"][0]) == case["L_star"]
        assert int(got["next_node"][0]) == case["next_node"]
        assert int(got["next_anchor"][0]) == case["next_anchor"]
        assert host(got["accepted"])[0][:case["L_star"] + 1].tolist() == case["accepted"]
        assert torch.equal(got["h_next"][0], hn[0, case["next_node"]])


# ---------------------------------------------------------------- failure detection

@cuda
def test_bounded_wait_reports_timeout_and_context_survives(S):
    """A pipeline wait that nothing satisfies gives up, reports
    SENSE_DEVST_TIMEOUT, and the device keeps working afterwards."""
    assert S.sense_device_status(clear=True) == 0
    t0 = __import__("time").perf_counter()
    bits_ = S.sense_selftest_timeout(100_000_000)  # ~50 ms of SM clocks
    assert bits_ & S.DEVST_TIMEOUT
    assert __import__("time").perf_counter() - t0 < 30
    dev = torch.device("cuda")
    keys = synth.clustered_unit_keys(2048, 128, 8, seed=1, device=dev)
    spans = synth.spans_uniform(2048, 4, 10, seed=1, device=dev)
    ds = S.sense_datastore_build(keys, spans)
    qs, _ = synth.noisy_queries(keys, 16, seed=1)
    sc, ix = S.sense_retrieve_topk(ds, qs, 8)
    torch.cuda.synchronize()
    assert S.sense_device_status(clear=True) == 0
    full = O.scores(bits(keys), bits(qs))
    for qi in range(16):
        check_topk(host(sc[qi]), host(ix[qi]), full[qi], 8)


# ---------------------------------------------------------------- drafting step in one call

@cuda
@pytest.mark.parametrize("n,d,m,q,k,cap,with_bits", [
    (50000, 512, 16, 1, 32, 64, True),      # the single-query path: one fused kernel
    (50000, 512, 16, 2, 128, 0, False),     # uncapped, 128 candidates
    (70000, 4096, 8, 4, 8, 10, True),       # cap below the node count
    (20000, 256, 32, 3, 64, 128, False),    # long spans
    (50000, 512, 16, 8, 32, 64, True),      # sampled-threshold retrieval (separate launches)
    (30000, 512, 16, 16, 64, 100, True),    # tensor-core retrieval (separate launches)
    (30000, 512, 4, 1, 200, 0, False),      # k > 128: the large trie (separate launches)
])
def test_draft_equals_separate_calls(S, n, d, m, q, k, cap, with_bits):
    """sense_draft is bit-identical to retrieve + gather + tree called one by
    one (which the other tests compare with the oracle), on every path."""
    dev = torch.device("cuda")
    keys = synth.clustered_unit_keys(n, d, 64, seed=n % 89, device=dev)
    spans = synth.spans_uniform(n, m, 6, seed=m, device=dev)  # few tokens: shared prefixes
    ds = S.sense_datastore_build(keys, spans)
    qs, _ = synth.noisy_queries(keys, q, seed=q + k)
    for _ in range(2):  # twice in a row: nothing left over from the first call matters
        got = S.sense_draft(ds, qs, k, node_cap=cap, mask_bits=with_bits)
        sc, ix = S.sense_retrieve_topk(ds, qs, k)
        dr = S.sense_gather_drafts(ds, ix)
        tr = S.sense_build_tree(dr, node_cap=cap, mask_bits=with_bits)
        torch.cuda.synchronize()
        assert S.sense_device_status(clear=True) == 0
        assert torch.equal(got["scores"], sc) and torch.equal(got["idx"], ix)
        assert torch.equal(got["spans"], dr)
        for key in ("num_nodes", "tokens", "parent", "depth", "gamma") + (("mask_bits",) if with_bits else ()):
            assert torch.equal(got[key], tr[key]), key
    full = O.scores(bits(keys), bits(qs))
    for qi in range(q):
        check_topk(host(got["scores"][qi]), host(got["idx"][qi]), full[qi], k)


@cuda
def test_prepared_calls_follow_buffer_contents(S):
    """A prepared call reissues the same call on the same buffers: after the
    query buffer's contents change, it gives what a fresh call gives."""
    dev = torch.device("cuda")
    n, d, m, q, k, cap, v = 30000, 512, 8, 1, 16, 32, 1000
    keys = synth.clustered_unit_keys(n, d, 64, seed=41, device=dev)
    spans = synth.spans_uniform(n, m, 6, seed=42, device=dev)
    ds = S.sense_datastore_build(keys, spans)
    qbuf = torch.empty(q, d, dtype=torch.bfloat16, device=dev)
    call, outs = S.sense_draft(ds, qbuf, k, node_cap=cap, prepare=True)
    root = synth.gate_logits(q, 1, v, seed=3, device=dev)[:, 0].contiguous()
    nodes = synth.gate_logits(q, cap, v, seed=4, device=dev)
    hr = synth.gate_hidden(q, 1, d, seed=3, device=dev)[:, 0].contiguous()
    hn = synth.gate_hidden(q, cap, d, seed=4, device=dev)
    gcall, gouts = S.sense_soft_gate(outs, root, nodes, hr, hn, prepare=True)
    for seed in (5, 6, 7):
        qs, _ = synth.noisy_queries(keys, q, seed=seed)
        qbuf.copy_(qs)
        call()
        gcall()
        want = S.sense_draft(ds, qs, k, node_cap=cap)
        wg = S.sense_soft_gate(want, root, nodes, hr, hn)
        torch.cuda.synchronize()
        assert S.sense_device_status(clear=True) == 0
        for key in ("scores", "idx", "spans", "num_nodes", "tokens", "parent", "gamma"):
            assert torch.equal(outs[key], want[key]), key
        for key in ("i_star", "L_star", "next_node", "next_anchor", "accepted", "h_next"):
            assert torch.equal(gouts[key], wg[key]), key


@cuda
def test_recorded_calls_follow_buffer_contents(S):
    """record_calls() marshals a step's calls once (retrieval, hybrid
    rerank with the dynamic buffer, trie, gate, R.Update): issuing them
    again on changed query contents gives what fresh calls give, and the
    recording itself runs nothing."""
    dev = torch.device("cuda")
    n, d, m, q, k, kd, cap, v = 30000, 512, 8, 1, 16, 8, 32, 1000
    keys = synth.clustered_unit_keys(n, d, 64, seed=51, device=dev)
    spans = synth.spans_uniform(n, m, 6, seed=52, device=dev)
    ds = S.sense_datastore_build(keys, spans)
    root = synth.gate_logits(q, 1, v, seed=3, device=dev)[:, 0].contiguous()
    nodes = synth.gate_logits(q, cap, v, seed=4, device=dev)
    hr = synth.gate_hidden(q, 1, d, seed=3, device=dev)[:, 0].contiguous()
    hn = synth.gate_hidden(q, cap, d, seed=4, device=dev)

    def step(ctx, query, anchor, outs):
        sc, ix = S.sense_retrieve_topk(ds, query, k, outs.get("sc"), outs.get("ix"),
                                       outs.get("ws"))
        outs["sc"], outs["ix"] = sc, ix
        dyn = S.sense_ctx_search(ctx, query, kd, 0.05, outs=outs.setdefault("dyn", {}),
                                 workspace=outs.get("dws"))
        dr = S.sense_hybrid_drafts(ds, sc, ix, dyn, anchor, k, True, out=outs.get("dr"))
        outs["dr"] = dr
        tr = S.sense_build_tree(dr, node_cap=cap, outs=outs.setdefault("tree", {}))
        g = S.sense_soft_gate(tr, root, nodes, hr, hn, outs=outs.setdefault("gate", {}),
                              workspace=outs.get("gws"))
        S.sense_ctx_append_path(ctx, hr[0], hn[0], tr["gamma"][0], g["i_star"][:1],
                                g["n_accept"][:1], g["accepted"][0])
        return outs

    def fresh_ctx():
        ctx = S.sense_ctx_create(256, d, m)
        rows = synth.gate_hidden(1, 40, d, seed=9, device=dev)[0].contiguous()
        S.sense_ctx_append(ctx, rows, torch.arange(40, dtype=torch.int32, device=dev))
        return ctx

    ctx_a, ctx_b = fresh_ctx(), fresh_ctx()
    qbuf = torch.zeros(q, d, dtype=torch.bfloat16, device=dev)
    anchor_a = torch.zeros(q, dtype=torch.int32, device=dev)
    outs_a = {"ws": S.alloc_workspace(S.sense_retrieve_workspace_bytes(ds, q, k), dev),
              "dws": S.alloc_workspace(S.lib().sense_ctx_search_workspace_bytes(
                  __import__("ctypes").c_void_p(ctx_a.handle), q, kd), dev),
              "gws": S.alloc_workspace(S.sense_soft_gate_workspace_bytes(q, cap, 3), dev)}
    before = ctx_a.count
    with S.record_calls() as calls:
        step(ctx_a, qbuf, anchor_a, outs_a)
    torch.cuda.synchronize()
    assert ctx_a.count == before and len(calls) == 6  # nothing ran
    anchor_b = torch.zeros(q, dtype=torch.int32, device=dev)
    for seed in (5, 6, 7):
        qs, _ = synth.noisy_queries(keys, q, seed=seed)
        qbuf.copy_(qs)
        for c in calls:
            c()
        want = step(ctx_b, qs, anchor_b, {})
        torch.cuda.synchronize()
        assert S.sense_device_status(clear=True) == 0
        for key in ("sc", "ix", "dr"):
            assert torch.equal(outs_a[key], want[key]), key
        for key in ("num_nodes", "tokens", "gamma"):
            assert torch.equal(outs_a["tree"][key], want["tree"][key]), key
        for key in ("i_star", "n_accept", "accepted", "next_anchor"):
            assert torch.equal(outs_a["gate"][key], want["gate"][key]), key
        assert ctx_a.count == ctx_b.count
