"""GPU-vs-oracle parity of the dynamic context buffer (R.Update, DynSearch
with the delta boost) and of the hybrid static + dynamic candidate list,
through the C ABI.  Inputs are seeded; expected values only from ``oracle``.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import ctx_oracle as X
from oracle import sense_oracle as O
from tests.parity import SCORE_TOL, bits, check_topk, host

pytestmark = pytest.mark.gpu
cuda = pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")


@pytest.fixture(scope="module")
def S():
    import paper_2606_00021_gb300 as S
    S.lib()
    return S


def _check_search(got, h_hist, tok_hist, cap, m, qb, k, delta):
    pos, keys, spans = X.ctx_entries(h_hist, tok_hist, cap, m)
    gp = host(got["pos"]).astype(np.int64)
    gs = host(got["scores"]).astype(np.float64)
    gsp = host(got["spans"])
    n_e = len(pos)
    row_of = {int(p): e for e, p in enumerate(pos)}
    full = O.scores(keys, qb) + delta if n_e else np.zeros((qb.shape[0], 0))
    for qi in range(qb.shape[0]):
        kk = min(k, n_e)
        assert (gp[qi, kk:] == -1).all() and np.isneginf(gs[qi, kk:]).all()
        assert (gsp[qi, kk:] == -1).all()
        if kk == 0:
            continue
        ent = np.array([row_of[int(p)] for p in gp[qi, :kk]])
        check_topk(gs[qi, :kk], ent, full[qi], kk)
        np.testing.assert_array_equal(gsp[qi, :kk], spans[ent])


@cuda
@pytest.mark.parametrize("cap,d,m,k,chunks", [
    (4096, 512, 16, 32, [100, 1, 3, 7, 16, 2]),
    (64, 256, 4, 8, [10, 30, 40, 5, 100, 1]),
    (40, 128, 8, 50, [3, 4, 5, 60]),
])
def test_ctx_append_and_search_match_oracle(S, cap, d, m, k, chunks):
    dev = torch.device("cuda")
    total = sum(chunks)
    h = synth.gaussian_rows_f32(total, d, seed=cap + d).to(torch.bfloat16)
    tok = torch.from_numpy(np.random.default_rng(m).integers(0, 1000, total).astype(np.int32))
    qs = synth.gaussian_rows_f32(3, d, seed=5).to(torch.bfloat16)
    hb, qb = bits(h), bits(qs)
    ctx = S.sense_ctx_create(cap, d, m)
    done = 0
    for c in chunks:
        S.sense_ctx_append(ctx, h[done:done + c].to(dev), tok[done:done + c].to(dev))
        done += c
        assert ctx.count == done
        got = S.sense_ctx_search(ctx, qs.to(dev), k, delta=0.5)
        torch.cuda.synchronize()
        assert S.sense_device_status(clear=True) == 0
        _check_search(got, hb[:done], tok.numpy()[:done], cap, m, qb, k, 0.5)
    ctx.reset()
    assert ctx.count == 0
    got = S.sense_ctx_search(ctx, qs.to(dev), k)
    assert (host(got["pos"]) == -1).all()
    ctx.close()


@cuda
def test_ctx_ties_bit_exact(S):
    """Basis-vector states: scores are exactly 0 or 1, so ties decide the
    order (older position first) and everything is compared bit for bit."""
    dev = torch.device("cuda")
    d, m, cap, T = 64, 3, 128, 90
    rng = np.random.default_rng(3)
    axis = rng.integers(0, 4, T)
    h = np.zeros((T, d), np.float32)
    h[np.arange(T), axis] = rng.choice([0.5, 2.0, 8.0], T)  # any positive scale
    hb = bits(torch.from_numpy(h).to(torch.bfloat16))
    tok = rng.integers(0, 50, T).astype(np.int32)
    q = np.zeros((4, d), np.float32)
    q[np.arange(4), np.arange(4)] = 1.0
    qb = bits(torch.from_numpy(q).to(torch.bfloat16))
    ctx = S.sense_ctx_create(cap, d, m)
    S.sense_ctx_append(ctx, torch.from_numpy(hb.view(np.int16)).view(torch.bfloat16).to(dev),
                       torch.from_numpy(tok).to(dev))
    got = S.sense_ctx_search(ctx, torch.from_numpy(qb.view(np.int16)).view(torch.bfloat16).to(dev),
                             40, delta=-0.25)
    torch.cuda.synchronize()
    ws, wp, wsp = X.ctx_search(hb, tok, cap, m, qb, 40, -0.25)
    np.testing.assert_array_equal(host(got["pos"]), wp)
    np.testing.assert_array_equal(host(got["scores"]), ws.astype(np.float32))
    np.testing.assert_array_equal(host(got["spans"]), wsp)


@cuda
@pytest.mark.parametrize("q,ks,kd,keep,anchored,force", [
    (4, 32, 16, 32, True, True), (3, 8, 8, 16, False, False), (2, 64, 0, 20, True, False),
    (5, 1, 40, 10, True, True), (2, 500, 300, 64, True, True),
])
def test_hybrid_drafts_match_oracle(S, q, ks, kd, keep, anchored, force):
    dev = torch.device("cuda")
    rng = np.random.default_rng(q * 100 + ks + kd)
    n, m = 5000, 6
    spans = synth.spans_uniform(n, m, 6, seed=ks).to(dev)
    s_idx = rng.integers(0, n, (q, ks)).astype(np.int32)
    # scores on a coarse grid so that ties across and within the lists occur
    s_sc = np.sort(rng.integers(0, 20, (q, ks)) / 16, axis=1)[:, ::-1].astype(np.float32).copy()
    d_sc = (np.sort(rng.integers(0, 20, (q, kd)) / 16, axis=1)[:, ::-1] + 0.25).astype(np.float32)
    if kd:
        d_sc[:, -max(1, kd // 4):] = -np.inf  # empty slots
    d_sp = rng.integers(0, 6, (q, kd, m)).astype(np.int32)
    anchor = rng.integers(0, 6, q).astype(np.int32) if anchored else None
    dyn = {"scores": torch.from_numpy(d_sc.copy()).to(dev),
           "spans": torch.from_numpy(d_sp).to(dev)} if kd else None
    ds = S.sense_datastore_build(torch.zeros(n, 8, dtype=torch.bfloat16, device=dev), spans)
    got = S.sense_hybrid_drafts(ds, torch.from_numpy(s_sc).to(dev), torch.from_numpy(s_idx).to(dev),
                                dyn, None if anchor is None else torch.from_numpy(anchor).to(dev),
                                keep, force)
    torch.cuda.synchronize()
    assert S.sense_device_status(clear=True) == 0
    sp_h = host(spans)
    want = X.hybrid_drafts(s_sc, sp_h[s_idx], d_sc if kd else np.zeros((q, 0)),
                           d_sp if kd else np.zeros((q, 0, m), np.int32), anchor, keep, force)
    np.testing.assert_array_equal(host(got), want)


def _path_case(rng, d, n_nodes, k, m):
    root = synth.gaussian_rows_f32(1, d, seed=int(rng.integers(1 << 30))).to(torch.bfloat16)[0]
    nodes = synth.gaussian_rows_f32(n_nodes, d, seed=int(rng.integers(1 << 30))).to(torch.bfloat16)
    gamma = rng.integers(0, n_nodes, (k, m)).astype(np.int32)
    accepted = rng.integers(0, 300, m).astype(np.int32)
    return root, nodes, gamma, accepted


@cuda
def test_ctx_append_path_matches_oracle(S):
    """R.Update of verified steps on the device: the appended history is the
    root state, then the states of the accepted path's nodes (through
    Gamma), with the accepted tokens; n_accept = 0 appends nothing."""
    dev = torch.device("cuda")
    rng = np.random.default_rng(21)
    d, m, cap, k, n_nodes = 256, 5, 64, 4, 20
    pre_h = synth.gaussian_rows_f32(10, d, seed=77).to(torch.bfloat16)
    pre_t = rng.integers(0, 300, 10).astype(np.int32)
    ctx = S.sense_ctx_create(cap, d, m)
    S.sense_ctx_append(ctx, pre_h.to(dev), torch.from_numpy(pre_t).to(dev))
    hist_h, hist_t = [bits(pre_h)], [pre_t]
    qs = synth.gaussian_rows_f32(2, d, seed=78).to(torch.bfloat16)
    for step, (i_star, n_acc) in enumerate([(2, 3), (0, 0), (3, 5), (1, 1), (2, 5)] * 4):
        root, nodes, gamma, acc = _path_case(rng, d, n_nodes, k, m)
        S.sense_ctx_append_path(ctx, root.to(dev), nodes.to(dev), torch.from_numpy(gamma).to(dev),
                                torch.tensor([i_star], dtype=torch.int32, device=dev),
                                torch.tensor([n_acc], dtype=torch.int32, device=dev),
                                torch.from_numpy(acc).to(dev))
        rows = [bits(root[None])[0]] + [bits(nodes[gamma[i_star, j - 1]][None])[0]
                                        for j in range(1, n_acc)]
        if n_acc:
            hist_h.append(np.stack(rows))
            hist_t.append(acc[:n_acc])
        got = S.sense_ctx_search(ctx, qs.to(dev), 12, delta=0.1)
        torch.cuda.synchronize()
        assert S.sense_device_status(clear=True) == 0
        hh, ht = np.concatenate(hist_h), np.concatenate(hist_t)
        assert ctx.count == len(ht)
        _check_search(got, hh, ht, cap, m, bits(qs), 12, 0.1)
    ctx.close()


@cuda
def test_ctx_step_replays_as_cuda_graph(S):
    """The device-side counter lets (append path, search) be captured once
    and replayed: each replay appends the accepted path again."""
    dev = torch.device("cuda")
    rng = np.random.default_rng(5)
    d, m, cap, k, n_nodes = 128, 4, 32, 3, 12
    root, nodes, gamma, acc = _path_case(rng, d, n_nodes, k, m)
    args = (root.to(dev), nodes.to(dev), torch.from_numpy(gamma).to(dev),
            torch.tensor([1], dtype=torch.int32, device=dev),
            torch.tensor([4], dtype=torch.int32, device=dev), torch.from_numpy(acc).to(dev))
    qs = synth.gaussian_rows_f32(2, d, seed=9).to(torch.bfloat16).to(dev)
    ctx = S.sense_ctx_create(cap, d, m)
    out = S.sense_ctx_search(ctx, qs, 6)  # outputs and workspace allocated before capture
    ws = S.alloc_workspace(S.lib().sense_ctx_search_workspace_bytes(
        __import__("ctypes").c_void_p(ctx.handle), 2, 6))
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        S.sense_ctx_append_path(ctx, *args)
        S.sense_ctx_search(ctx, qs, 6, outs=out, workspace=ws)
    ctx.reset()
    rows = np.stack([bits(root[None])[0]] + [bits(nodes[gamma[1, j - 1]][None])[0]
                                             for j in range(1, 4)])
    for rep in range(1, 4):
        g.replay()
        torch.cuda.synchronize()
        assert ctx.count == 4 * rep
        hh = np.concatenate([rows] * rep)
        ht = np.concatenate([acc[:4]] * rep)
        _check_search(out, hh, ht, cap, m, bits(qs.cpu()), 6, 0.0)
    ctx.close()


@cuda
@pytest.mark.parametrize("cap,m,fill,ks,kd,keep,force,node_cap,q", [
    (4096, 16, 3000, 32, 16, 32, True, 64, 1),     # the bench's shape: fused tail
    (256, 8, 30, 20, 30, 40, False, 0, 2),         # fewer searchable entries than kd
    (512, 4, 600, 8, 8, 10, True, 7, 3),           # ring wrapped, tight node cap
    (128, 8, 100, 100, 60, 150, False, 0, 1),      # n_keep > 128: the calls one by one
])
def test_dyn_draft_equals_separate_calls(S, cap, m, fill, ks, kd, keep, force, node_cap, q):
    """sense_dyn_draft is bit-identical to sense_ctx_search, then
    sense_hybrid_drafts, then sense_build_tree (with mask bits), in its
    fused form (n_keep <= 128) and in its fallback."""
    dev = torch.device("cuda")
    d, n = 256, 5000
    keys = synth.clustered_unit_keys(n, d, 16, seed=cap + ks, device=dev)
    spans = synth.spans_uniform(n, m, 7, seed=m, device=dev)  # small vocab: shared prefixes
    ds = S.sense_datastore_build(keys, spans)
    ctx = S.sense_ctx_create(cap, d, m)
    h = synth.gaussian_rows_f32(fill, d, seed=fill).to(torch.bfloat16).to(dev)
    tok = torch.from_numpy(np.random.default_rng(fill).integers(0, 7, fill).astype(np.int32))
    S.sense_ctx_append(ctx, h, tok.to(dev))
    qs, _ = synth.noisy_queries(keys, q, seed=3)
    sc, ix = S.sense_retrieve_topk(ds, qs, ks)
    anchor = torch.from_numpy(np.arange(q, dtype=np.int32) % 7).to(dev)
    for _ in range(2):
        got = S.sense_dyn_draft(ds, ctx, qs, sc, ix, kd, delta=0.05, anchor=anchor,
                                n_keep=keep, force_anchor=force, node_cap=node_cap,
                                mask_bits=True)
        dyn = S.sense_ctx_search(ctx, qs, kd, 0.05)
        dr = S.sense_hybrid_drafts(ds, sc, ix, dyn, anchor, keep, force)
        tr = S.sense_build_tree(dr, node_cap=node_cap, mask_bits=True)
        torch.cuda.synchronize()
        assert S.sense_device_status(clear=True) == 0
        for key in ("scores", "pos", "spans"):
            assert torch.equal(got["dyn"][key], dyn[key]), key
        assert torch.equal(got["spans"], dr)
        for key in ("num_nodes", "tokens", "parent", "depth", "gamma", "mask_bits"):
            assert torch.equal(got[key], tr[key]), key
