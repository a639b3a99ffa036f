"""Benchmark of the SENSE drafting hot path on GB300.

One step = one pass of the whole path for one batch of queries on a seeded
synthetic workload resident in HBM: exact top-k retrieval over the bf16
datastore, span gather, loose-trie draft tree and soft-gated evaluation.

Default workload (LLaMA-70B-shaped store, the largest that one GPU holds):
n = 8,388,608 keys, d = 8192 bf16 (137 GB), 1 query per step (16 distinct
queries, each a perturbed key), k = 64, spans of 16 Zipf(1.1) tokens over a
128,256-token vocabulary, tree capped at 64 nodes, gate on fp32 N(0, 3^2)
logits for every tree node with the paper's defaults (gamma 0.05, top-3,
window 6).  ``--workload`` selects the other shapes (llama7b_1m, qwen7b_4m,
the sweeps, tiny_4k).

Prints one JSON line (rank 0).  ``--impl reference`` times the CPU oracle
on bounded samples of the same workload instead.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

import synth  # noqa: E402
from synth.workloads import WORKLOADS  # noqa: E402

DEFAULT = "llama70b_8m"
METRIC = "hidden-state top-k retrieval queries/s (whole drafting step)"
GATE = dict(gamma=0.05, topk=3, window=6, tau=0)
# DRAM bytes (read + write) per unit processed by the dominant kernels, each
# from one ncu capture of a smaller case of the same kernel and shape (the
# summaries in profiles/), scaled in the bench line by the units of a full
# step: key rows for the scans (keyed by d), logits rows for the gate's row
# pass (keyed by V).  Traffic grows in proportion to those units.
NCU_TRAFFIC_PER_UNIT = {
    # 262,144 x 4096 keys: 2,147,567,104 B read + 2,790,912 B written
    ("scan_gemv", 4096): (2147567104 + 2790912) / 262144,
    # 262,144 x 8192 keys: 4,295,055,872 B read + 2,958,336 B written
    ("scan_gemv", 8192): (4295055872 + 2958336) / 262144,
    # 524,288 x 3584 keys, sample + rest launches of one step (two slices
    # per ring stage)
    ("scan_tc", 3584): (235059200 + 3039488 + 3523413504 + 171008) / 524288,
    # 4 queries of the k = 64 sweep: 3,774 root / inner-node rows of 128,256 logits
    ("gate_rows", 128256): (1939918336 + 3338240) / 3773.9375,
}


def _bits(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor -> uint16 bit patterns on the host."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def _host(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().numpy()


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            j = json.load(f)
        return float(j["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """Samples SM clocks and throttle reasons with nvidia-smi while running."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out = ""
        sms, maxs, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sms.append(float(parts[0]))
                maxs.append(float(parts[1]))
            except ValueError:
                continue
            for name, val in zip(names, parts[4:8]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sms:
            return None
        return {"sm_mhz": statistics.median(sms), "sm_max_mhz": max(maxs),
                "reasons": sorted(reasons), "samples": len(sms)}


def max_over_ranks(x: float, dist=None, device="cpu") -> float:
    """The largest of every rank's value (timings are taken as the slowest)."""
    if dist is None:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: int, world: int, seconds: float) -> float:
    """Whole-job units per second: every rank processed units_per_rank."""
    return world * units_per_rank / seconds


def make_workload(cfg, dev, seed=0, key_recipe=None):
    import synth
    n, d, m = cfg["n"], cfg["d"], cfg["m"]
    if key_recipe and key_recipe.get("kind") == "subspace":
        keys, assign = synth.subspace_unit_keys(n, d, cfg["clusters"], rank=key_recipe["rank"],
                                                decay=key_recipe["decay"], sigma=0.3,
                                                iso=key_recipe["iso"], seed=seed, device=dev,
                                                return_assign=True)
    else:
        keys, assign = synth.clustered_unit_keys(n, d, cfg["clusters"], sigma=0.3, seed=seed,
                                                 device=dev, return_assign=True)
    if cfg["zipf"]:
        spans = synth.spans_zipf(n, m, cfg["vocab"], 1.1, seed=seed, device=dev)
    else:
        spans = synth.spans_uniform(n, m, cfg["vocab"], seed=seed, device=dev)
    n_q = cfg["distinct"] * cfg["q"]
    queries, src = synth.noisy_queries(keys, n_q, noise=0.05, seed=seed + 1)
    queries = queries.reshape(cfg["distinct"], cfg["q"], d).contiguous()
    return keys, spans, queries, assign


def make_gate_inputs(cfg, dev, sets=4, seed=0):
    import synth
    q, k, m = cfg["q"], cfg["k"], cfg["m"]
    cap = cfg["cap"] if cfg["cap"] > 0 else k * m
    out = []
    for s in range(sets):
        root = synth.gate_logits(q, 1, cfg["vocab"], seed=seed + 10 * s, device=dev)[:, 0].contiguous()
        nodes = synth.gate_logits(q, cap, cfg["vocab"], seed=seed + 10 * s + 1, device=dev)
        hr = synth.gate_hidden(q, 1, cfg["d"], seed=seed + 10 * s, device=dev)[:, 0].contiguous()
        hn = synth.gate_hidden(q, cap, cfg["d"], seed=seed + 10 * s + 1, device=dev)
        out.append((root, nodes, hr, hn))
    return out


class Pipeline:
    """Preallocated buffers and one step of the path through the C ABI."""

    def __init__(self, S, ds, cfg, dev):
        self.S, self.ds, self.cfg = S, ds, cfg
        q, k, m = cfg["q"], cfg["k"], cfg["m"]
        self.cap = cfg["cap"] if cfg["cap"] > 0 else k * m
        self.scores = torch.empty(q, k, dtype=torch.float32, device=dev)
        self.idx = torch.empty(q, k, dtype=torch.int32, device=dev)
        self.ws = S.alloc_workspace(S.sense_retrieve_workspace_bytes(ds, q, k), dev)
        self.drafts = torch.empty(q, k, m, dtype=torch.int32, device=dev)
        self.tree = {}
        self.gate = {}
        self.ann = None
        self.gws = S.alloc_workspace(S.sense_soft_gate_workspace_bytes(q, self.cap, GATE["topk"]), dev)

    def use_ann(self, ann, dev):
        """Retrieve through the projected IVF index instead of the exact scan;
        with ann["rerank"] = N' > 0 the index returns N' candidates whose exact
        similarity to the full query ranks them (Eq. 8's sim) before the top k
        are kept."""
        q, k = self.cfg["q"], self.cfg["k"]
        self.ann = ann
        kk = max(k, ann.get("rerank", 0))
        self.qproj = torch.empty(q, ann["index"].v, dtype=torch.float32, device=dev)
        if ann.get("rerank", 0):
            self.cand_s = torch.empty(q, kk, dtype=torch.float32, device=dev)
            self.cand_i = torch.empty(q, kk, dtype=torch.int32, device=dev)
        self.ws = self.S.alloc_workspace(
            self.S.sense_ivf_search_workspace_bytes(ann["index"], q, kk, ann["nprobe"]), dev)
        import ctypes
        self.ann_ws = self.S.alloc_workspace(self.S.lib().sense_ann_draft_workspace_bytes(
            ctypes.c_void_p(ann["index"].handle), q, k, ann["nprobe"], ann.get("rerank", 0)), dev)

    def retrieve(self, query):
        S, cfg = self.S, self.cfg
        if self.ann is None:
            S.sense_retrieve_topk(self.ds, query, cfg["k"], self.scores, self.idx, self.ws)
        else:  # projection, search (and re-scoring) in one call
            a = self.ann
            S.sense_ann_search(a["index"], self.ds, query, a["basis"], a["mean"], cfg["k"],
                               a["nprobe"], rerank=a.get("rerank", 0), out_scores=self.scores,
                               out_idx=self.idx, workspace=self.ann_ws)

    def use_dynamic(self, ctx, kd, delta, dev):
        """Hybrid retrieval (Alg. 2): the dynamic buffer is searched beside the
        static store, the union is reranked with the previous step's anchor,
        and the accepted path is appended after the gate (Alg. 1 R.Update)."""
        q = self.cfg["q"]
        self.dyn = {"ctx": ctx, "kd": kd, "delta": delta, "outs": {},
                    "ws": self.S.alloc_workspace(self.S.lib().sense_ctx_search_workspace_bytes(
                        __import__("ctypes").c_void_p(ctx.handle), q, kd), dev)}
        # x~ of the next step: the gate writes it, the next step's rerank reads it
        self.gate["next_anchor"] = torch.zeros(q, dtype=torch.int32, device=dev)

    def use_verify(self, heads, prefix, dev, seed=0):
        """Adds the tree-masked attention of the verify forward (Alg. 1) on a
        synthetic KV cache: heads x 128-dim, `prefix` committed positions,
        the tree's cap rows as draft tokens."""
        L = self.cap
        capacity = ((prefix + L + 127) // 128) * 128
        g = torch.Generator(device=dev).manual_seed(seed + 21)
        mk = lambda *shape: torch.randn(*shape, generator=g, device=dev).to(torch.bfloat16)
        self.verify = {"q": mk(heads, L, 128), "k": mk(heads, capacity, 128),
                       "vt": mk(heads, 128, capacity), "prefix": prefix,
                       "scale": 1.0 / 128 ** 0.5,
                       "out": torch.empty(heads, L, 128, dtype=torch.float32, device=dev),
                       "ws": self.S.alloc_workspace(self.S.lib().sense_tree_attention_workspace_bytes(
                           heads, L, prefix), dev),
                       "heads": heads, "L": L, "capacity": capacity}

    def invalidate(self):
        """Forget the prepared calls (their output buffers were replaced)."""
        self._calls = {}

    def _prepared(self, key, make):
        calls = self.__dict__.setdefault("_calls", {})
        c = calls.get(key)
        if c is None:
            c = calls[key] = make()
        return c

    def step(self, query, gate_in, before_gate=None):
        S, cfg = self.S, self.cfg
        dyn = getattr(self, "dyn", None)
        ver = getattr(self, "verify", None)
        if dyn is None and ver is None:
            # the step's two library calls, marshalled once per (query,
            # gate-input) buffer and issued again every step
            def make_draft():
                outs = self.tree
                outs["scores"], outs["idx"], outs["spans"] = self.scores, self.idx, self.drafts
                if self.ann is None:
                    call, _ = S.sense_draft(self.ds, query, cfg["k"], node_cap=cfg["cap"],
                                            outs=outs, workspace=self.ws, prepare=True)
                else:
                    a = self.ann
                    call, _ = S.sense_ann_draft(a["index"], self.ds, query, a["basis"], a["mean"],
                                                cfg["k"], a["nprobe"], rerank=a.get("rerank", 0),
                                                node_cap=cfg["cap"], outs=outs,
                                                workspace=self.ann_ws, prepare=True)
                return call

            def make_gate():
                root, nodes, hr, hn = gate_in
                call, _ = S.sense_soft_gate(self.tree, root, nodes, hr, hn, workspace=self.gws,
                                            outs=self.gate, prepare=True, **GATE)
                return call

            stream = S._stream(None)  # calls captured into a graph run on another stream
            self._prepared(("draft", stream, query.data_ptr()), make_draft)()
            if before_gate is not None:
                before_gate()
            self._prepared(("gate", stream) + tuple(t.data_ptr() for t in gate_in), make_gate)()
            return
        # with the dynamic buffer or the verify attention: the step's calls,
        # recorded once per buffer set (arguments marshalled once) and issued
        # again every step
        def make_pre():
            with S.record_calls() as calls:
                if dyn is None:
                    # retrieval, gather and trie in one call (exact: one kernel
                    # per query after the scan on the single-pass path)
                    outs = self.tree
                    outs["scores"], outs["idx"], outs["spans"] = self.scores, self.idx, self.drafts
                    if self.ann is None:
                        S.sense_draft(self.ds, query, cfg["k"], node_cap=cfg["cap"],
                                      mask_bits=ver is not None, outs=outs, workspace=self.ws)
                    else:
                        a = self.ann
                        S.sense_ann_draft(a["index"], self.ds, query, a["basis"], a["mean"],
                                          cfg["k"], a["nprobe"], rerank=a.get("rerank", 0),
                                          node_cap=cfg["cap"], mask_bits=ver is not None,
                                          outs=outs, workspace=self.ann_ws)
                else:
                    # static retrieval, then DynSearch, the hybrid rerank and the
                    # trie in one call
                    self.retrieve(query)
                    outs = self.tree
                    outs["dyn"], outs["spans"] = dyn["outs"], self.drafts
                    S.sense_dyn_draft(self.ds, dyn["ctx"], query, self.scores, self.idx,
                                      dyn["kd"], dyn["delta"], self.gate["next_anchor"],
                                      cfg["k"], True, node_cap=cfg["cap"],
                                      mask_bits=ver is not None, outs=outs,
                                      workspace=dyn["ws"])
                if ver is not None:
                    S.sense_tree_attention(ver["q"], ver["k"], ver["vt"], ver["prefix"],
                                           self.tree["mask_bits"][0], ver["scale"], out=ver["out"],
                                           workspace=ver["ws"])
            return calls

        def make_post():
            root, nodes, hr, hn = gate_in
            with S.record_calls() as calls:
                S.sense_soft_gate(self.tree, root, nodes, hr, hn, workspace=self.gws,
                                  outs=self.gate, **GATE)
                if dyn is not None:  # R.Update with the accepted path
                    g = self.gate
                    S.sense_ctx_append_path(dyn["ctx"], hr[0], hn[0], self.tree["gamma"][0],
                                            g["i_star"][:1], g["n_accept"][:1], g["accepted"][0])
            return calls

        stream = S._stream(None)
        for c in self._prepared(("pre", stream, query.data_ptr()), make_pre):
            c()
        if before_gate is not None:
            before_gate()
        for c in self._prepared(("post", stream) + tuple(t.data_ptr() for t in gate_in), make_post):
            c()


DRAFT_KERNELS = ("scan_gemv", "scan_tc", "threshold", "merge", "pad_queries", "gather", "tree",
                 "project", "ivf_coarse", "ivf_scan", "ctx", "rescore", "draft")


def draft_kernel_rate(prof, q, tokens_per_query, steps):
    """tokens per query x queries / summed time of the drafting kernels."""
    ms = sum(prof.get(name, (0.0, 0))[0] for name in DRAFT_KERNELS)
    return q * tokens_per_query * steps / (ms / 1e3) if ms > 0 else None


class GraphStep:
    """The whole drafting step captured as one CUDA graph per gate-input set.
    The graphs read the query from a fixed staging buffer; a step copies the
    next query into it (device to device) and replays one graph."""

    def __init__(self, pipe, query0, gate_sets):
        self.d_query = torch.empty_like(query0)
        self.d_query.copy_(query0)
        self.graphs = []
        for gset in gate_sets:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                pipe.step(self.d_query, gset)
            self.graphs.append(g)
        torch.cuda.synchronize()

    def step(self, query, gi):
        self.d_query.copy_(query, non_blocking=True)
        self.graphs[gi].replay()


def build_ann(S, keys, kind, nlist, nprobe, pq_m, v, dev, seed=0):
    """Index construction for the approximate path (outside the timed region):
    the PCA basis is fitted offline on a 65,536-key sample (top eigenvectors
    of its covariance, by scipy on the host, as the paper's setup fits PCA
    with a library); keys are
    projected and normalised, the coarse quantizer is trained by spherical
    k-means (10 rounds on 64 x nlist keys), PQ codebooks by k-means on the
    residual sub-vectors (10 rounds), and the index is built - all but the
    PCA fit in the library's kernels."""
    n, d = keys.shape
    g = torch.Generator(device=dev).manual_seed(seed + 7)
    sample = keys[torch.randint(0, n, (min(n, 65536),), generator=g, device=dev)].float()
    mean = sample.mean(0)
    xc = sample - mean
    cov = (xc.T @ xc / xc.shape[0]).double().cpu().numpy()
    del sample, xc
    import scipy.linalg
    evals, evecs = scipy.linalg.eigh(cov, subset_by_index=[d - v, d - 1])
    energy = float(evals.sum() / np.trace(cov))  # variance kept by the v components
    basis = torch.from_numpy(np.ascontiguousarray(evecs[:, ::-1].T)).float().to(dev).contiguous()
    mean = mean.contiguous()
    del cov, evecs
    t0 = time.perf_counter()
    kp = torch.empty(n, v, dtype=torch.float32, device=dev)
    for lo in range(0, n, 1 << 20):
        hi = min(n, lo + (1 << 20))
        S.sense_project(keys[lo:hi], basis, mean, out=kp[lo:hi])
    train = kp[torch.randperm(n, generator=g, device=dev)[:min(n, 64 * nlist)]].contiguous()
    cent = S.sense_kmeans(train, train[:nlist].clone(), 10, True)
    cbs = None
    if kind == "ivfpq":
        _, res = S.sense_ivf_residuals(train, cent)
        dsub = v // pq_m
        cbs = torch.stack([S.sense_kmeans(res[:, m * dsub:(m + 1) * dsub],
                                          res[:256, m * dsub:(m + 1) * dsub].contiguous(), 10,
                                          False) for m in range(pq_m)])
        del res
    ix = S.sense_ivf_build(kp, cent, cbs)
    torch.cuda.synchronize()
    build_s = time.perf_counter() - t0
    sizes = (ix.arrays()["offsets"][1:] - ix.arrays()["offsets"][:-1]).float()
    del train
    return {"index": ix, "basis": basis, "mean": mean, "nprobe": nprobe, "kind": kind,
            "keys_proj": kp,
            "nlist": nlist, "pq_m": pq_m if kind == "ivfpq" else 0, "v": v,
            "pca_energy": energy,
            "build_s": build_s, "mean_list": float(sizes.mean()), "max_list": ix.max_list}


SLICE_ROWS = 65536  # rows per sampled slice of the store (one generator chunk)
REF_BUDGET_S = 150.0  # --impl reference: oracle time of the whole run, about


def _oracle_query(O, cfg, kb_slices, row_ids, qb, spans_h, gate_h):
    """One query batch through the oracle over the sampled rows: scoring and
    top-k over the sample (timed together), then gather, trie and gate on
    the sample's top-k (timed apart).  Returns (t_scan, t_down)."""
    t0 = time.perf_counter()
    s = np.concatenate([O.scores(kb, qb) for kb in kb_slices], axis=1)
    _, pos = O.topk(s, cfg["k"])
    t1 = time.perf_counter()
    idx = row_ids[pos]
    dr = O.gather_drafts(spans_h, idx)
    tr = O.loose_trie(dr, node_cap=cfg["cap"])
    root, nodes, hr, hn = gate_h
    O.soft_gate(tr["tokens"], tr["parent"], tr["num_nodes"], tr["gamma"], root, nodes, hr, hn,
                gamma_thr=GATE["gamma"], kappa=GATE["topk"], window=GATE["window"])
    return t1 - t0, time.perf_counter() - t1


def _gate_host(gate_set):
    return [_bits(t) if t.dtype == torch.bfloat16 else _host(t) for t in gate_set]


def cpu_baseline(cfg, keys, spans, queries, gate_sets, budget_s=10.0):
    """The oracle, as it stands, on whole queries of the same workload.

    Scoring and top-k run over seeded 65,536-row slices of the resident store,
    copied to the host one at a time, until about ``budget_s`` of oracle time
    is spent (the whole store when it fits); their time is scaled by
    n / rows scanned.  Gather, trie and gate run on the sample's top-k and
    are not scaled."""
    import oracle as O
    n = cfg["n"]
    n_slices = (n + SLICE_ROWS - 1) // SLICE_ROWS
    order = np.random.default_rng(5).permutation(n_slices)
    qb = _bits(queries[0])
    spans_h = _host(spans)
    gate_h = _gate_host(gate_sets[0])
    # the rate of the first slice sizes the sample to the budget
    lo0 = int(order[0]) * SLICE_ROWS
    kb0 = _bits(keys[lo0:min(n, lo0 + SLICE_ROWS)])
    t0 = time.perf_counter()
    O.scores(kb0, qb)
    take = int(min(n_slices, max(1, budget_s / max(time.perf_counter() - t0, 1e-6))))
    kbs, ids, rows = [], [], 0
    for si in order[:take]:
        lo, hi = int(si) * SLICE_ROWS, min(n, (int(si) + 1) * SLICE_ROWS)
        kbs.append(kb0 if lo == lo0 else _bits(keys[lo:hi]))
        ids.append(np.arange(lo, hi))
        rows += hi - lo
    # one whole query over the sample, timed end to end
    t_scan, t_down = _oracle_query(O, cfg, kbs, np.concatenate(ids), qb, spans_h, gate_h)
    scale = n / rows
    per_batch = t_scan * scale + t_down
    q = cfg["q"]
    return {"value": q / per_batch, "unit": "queries/s", "cores": os.cpu_count(),
            "kind": "oracle",
            "sample": (f"1 batch of {q} query(ies): oracle scoring + top-k over {rows} of {n} "
                       f"keys ({len(kbs)} seeded {SLICE_ROWS}-row slices copied from the device; "
                       f"{t_scan:.2f} s, scaled by n/rows = {scale:.2f}), then gather/trie/gate "
                       f"on that top-k ({t_down:.2f} s, unscaled); numpy fp64")}


def run_reference(args, cfg, name):
    """--impl reference: the CPU oracle on bounded samples of the same
    workload, one query batch per step.

    The store is not held: a pool of seeded 65,536-row slices of it (the
    generator's own chunks, drawn on the GPU when there is one, so the values
    are the main arm's), including the chunks of the step queries' source
    keys, is made before the timed steps.  Each step scores its query batch
    against ``--ref-slices`` slices of the pool (rotating), takes the top-k of
    that sample and runs gather, trie and gate on it; that is the step the
    line's ms_per_step times.  queries/s scales the scoring + top-k time by
    n / rows scanned (the full store), the rest unscaled."""
    import oracle as O
    import synth
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    n, d, q = cfg["n"], cfg["d"], cfg["q"]
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    store = synth.ClusteredStoreRows(n, d, cfg["clusters"], sigma=0.3, seed=0, device=dev)
    n_q = cfg["distinct"] * q
    queries, src = synth.noisy_queries(store, n_q, noise=0.05, seed=1)
    queries = queries.reshape(cfg["distinct"], q, d)
    src = src.reshape(cfg["distinct"], q).cpu()
    n_chunks = (n + synth.CHUNK_ROWS - 1) // synth.CHUNK_ROWS
    per_step = max(1, min(args.ref_slices, n_chunks))
    pool_ids = sorted(set((src[0] // synth.CHUNK_ROWS).tolist()))
    rng = np.random.default_rng(3)
    for c in rng.permutation(n_chunks).tolist():
        if len(pool_ids) >= min(n_chunks, 2 * per_step):
            break
        if c not in pool_ids:
            pool_ids.append(c)
    pool = {c: _bits(store.chunk(c)) for c in pool_ids}
    if cfg["zipf"]:
        spans = synth.spans_zipf(n, cfg["m"], cfg["vocab"], 1.1, seed=0, device=dev)
    else:
        spans = synth.spans_uniform(n, cfg["m"], cfg["vocab"], seed=0, device=dev)
    spans_h = _host(spans)
    del spans, store
    gate_h = _gate_host(make_gate_inputs(cfg, dev, sets=1, seed=100)[0])
    total = args.warmup + args.steps
    # rows per step: --ref-slices slices, fewer when the whole run would
    # exceed about REF_BUDGET_S (one untimed calibration step sizes it)
    c0 = pool_ids[0]
    ts1, td1 = _oracle_query(O, cfg, [pool[c0]], np.arange(c0 * synth.CHUNK_ROWS,
                                                           c0 * synth.CHUNK_ROWS + pool[c0].shape[0]),
                             _bits(queries[0]), spans_h, gate_h)
    per_row = ts1 / pool[c0].shape[0]
    step_budget = REF_BUDGET_S / total
    rows_cap = per_step * SLICE_ROWS
    rows_step = int(min(rows_cap, max(4096, (step_budget - td1) / max(per_row, 1e-12))))
    t_scan, t_down, t_step, rows_per = [], [], [], []
    for it in range(total):
        ids = [pool_ids[(it * per_step + j) % len(pool_ids)] for j in range(per_step)]
        kbs, row_ids, left = [], [], rows_step
        for c in ids:
            if left <= 0:
                break
            r = min(left, pool[c].shape[0])
            kbs.append(pool[c][:r])
            row_ids.append(np.arange(c * synth.CHUNK_ROWS, c * synth.CHUNK_ROWS + r))
            left -= r
        row_ids = np.concatenate(row_ids)
        qb = _bits(queries[it % cfg["distinct"]])
        t0 = time.perf_counter()
        ts, td = _oracle_query(O, cfg, kbs, row_ids, qb, spans_h, gate_h)
        el = time.perf_counter() - t0
        if it >= args.warmup:
            t_scan.append(ts)
            t_down.append(td)
            t_step.append(el)
            rows_per.append(row_ids.size)
    rows = statistics.mean(rows_per)
    scale = n / rows
    per_batch = statistics.mean(t_scan) * scale + statistics.mean(t_down)
    value = q / per_batch
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "queries/s",
        "n_gpus": args.gpus, "steps": len(t_step), "warmup": args.warmup,
        "ms_per_step": statistics.mean(t_step) * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": name, **{k: cfg[k] for k in ("n", "d", "q", "k", "m", "vocab",
                                                             "cap", "clusters")}},
        "cpu_baseline": {"value": value, "unit": "queries/s", "cores": os.cpu_count(),
                         "kind": "oracle",
                         "sample": (f"per step: one batch of {q} query(ies) of the workload "
                                    f"scored against {int(rows)} of its {n} keys (seeded "
                                    f"{SLICE_ROWS}-row slices of the store, at most "
                                    f"{per_step}, fewer rows when {total} steps would exceed "
                                    f"~{REF_BUDGET_S:.0f} s), top-k of that sample, "
                                    f"gather/trie/gate; ms_per_step is that sampled step; "
                                    f"value scales scoring + top-k by n/rows = {scale:.1f}; "
                                    f"numpy fp64"),
                         "scan_s_per_step": statistics.mean(t_scan),
                         "downstream_s_per_step": statistics.mean(t_down)},
        "e2e": {"value": value, "unit": "queries/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="sense", choices=["sense", "reference"])
    ap.add_argument("--workload", default=DEFAULT, choices=sorted(WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--ref-slices", type=int, default=4,
                    help="--impl reference: 65,536-row slices of the store scored per step")
    ap.add_argument("--e2e-steps", type=int, default=200)
    ap.add_argument("--n-keys", type=int, default=0,
                    help="override the store size (small cases for profiler captures)")
    ap.add_argument("--queries", type=int, default=0,
                    help="override the queries per step (small cases for profiler captures)")
    ap.add_argument("--retrieval", default="exact", choices=["exact", "ivfpq", "ivfflat"],
                    help="exact scan of the full keys, or the PCA + IVF index of App. E")
    ap.add_argument("--keys", default="clustered", choices=["clustered", "subspace"],
                    help="key recipe: isotropic clusters in d dimensions, or clusters and "
                         "spread inside a low-dimensional subspace (power-law spectrum)")
    ap.add_argument("--key-rank", type=int, default=256)
    ap.add_argument("--key-decay", type=float, default=1.0)
    ap.add_argument("--key-iso", type=float, default=0.05)
    ap.add_argument("--rerank", type=int, default=0, metavar="N_PRIME",
                    help="approximate retrieval: take N' candidates from the index and keep "
                         "the top k by their exact similarity to the full query (Eq. 8)")
    ap.add_argument("--nlist", type=int, default=4096)
    ap.add_argument("--nprobe", type=int, default=32)
    ap.add_argument("--pq-m", type=int, default=16)
    ap.add_argument("--proj-dim", type=int, default=64)
    ap.add_argument("--graph", action="store_true",
                    help="time CUDA graph replays of the whole step (per-kernel times then "
                         "come from an eager pass after the timed region)")
    ap.add_argument("--no-graph-line", action="store_true",
                    help="skip the supplementary graph-replay measurement of an eager run")
    ap.add_argument("--dynamic", type=int, default=0, metavar="CAPACITY",
                    help="add the dynamic context buffer of this many positions (q = 1)")
    ap.add_argument("--verify", type=int, default=0, metavar="HEADS",
                    help="add the tree-masked verify attention on a synthetic KV cache (q = 1)")
    ap.add_argument("--verify-prefix", type=int, default=4096)
    ap.add_argument("--dyn-k", type=int, default=16)
    ap.add_argument("--delta", type=float, default=0.05)
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    cfg = dict(WORKLOADS[args.workload])
    if args.n_keys > 0:
        cfg["n"] = args.n_keys
        args.workload = f"{args.workload}@n={args.n_keys}"
    if args.queries > 0:
        cfg["q"] = args.queries
        args.workload = f"{args.workload}@q={args.queries}"
    if args.impl == "reference":
        run_reference(args, cfg, args.workload)
        return

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    import paper_2606_00021_gb300 as S
    from paper_2606_00021_gb300 import _build
    _build.build()
    S.lib()

    key_recipe = ({"kind": "subspace", "rank": args.key_rank, "decay": args.key_decay,
                   "iso": args.key_iso} if args.keys == "subspace" else {"kind": "clustered"})
    keys, spans, queries, assign = make_workload(cfg, dev, seed=rank, key_recipe=key_recipe)
    cap = cfg["cap"] if cfg["cap"] > 0 else cfg["k"] * cfg["m"]
    gate_bytes = cfg["q"] * (cap + 1) * cfg["vocab"] * 4
    n_sets = 4 if gate_bytes < (2 << 30) else 1
    gate_sets = make_gate_inputs(cfg, dev, sets=n_sets, seed=100 + rank)
    ds = S.sense_datastore_build(keys, spans)
    pipe = Pipeline(S, ds, cfg, dev)
    nq = queries.shape[0]
    ann = None
    if args.retrieval != "exact":
        ann = build_ann(S, keys, args.retrieval, args.nlist, args.nprobe, args.pq_m,
                        args.proj_dim, dev, seed=rank)
        ann["rerank"] = args.rerank
        pipe.use_ann(ann, dev)
    if args.verify:
        if cfg["q"] != 1 or pipe.cap > 128:
            raise SystemExit("--verify models one sequence with at most 128 tree nodes")
        pipe.use_verify(args.verify, args.verify_prefix, dev, seed=rank)
    dyn_info = None
    if args.dynamic:
        if cfg["q"] != 1:
            raise SystemExit("--dynamic models one sequence: use a workload with q = 1")
        # prefill: the buffer starts full of the sequence's own states (store
        # keys of random clusters stand in for them) and Zipf tokens
        ctx = S.sense_ctx_create(args.dynamic, cfg["d"], cfg["m"])
        g = torch.Generator(device=dev).manual_seed(rank + 11)
        pre = keys[torch.randint(0, cfg["n"], (args.dynamic,), generator=g, device=dev)]
        pre_tok = synth.spans_zipf(args.dynamic, 1, cfg["vocab"], 1.1, seed=rank + 12,
                                   device=dev)[:, 0].contiguous()
        S.sense_ctx_append(ctx, pre.contiguous(), pre_tok)
        del pre
        pipe.use_dynamic(ctx, args.dyn_k, args.delta, dev)
        dyn_info = {"capacity": args.dynamic, "prefill": args.dynamic, "k_dynamic": args.dyn_k,
                    "delta": args.delta, "n_keep": cfg["k"], "anchor": "previous step's x~",
                    "update": "accepted path appended every step (device-side count)"}

    # warm-up, profiled: the kernel family with the largest share is the one
    # the timed region brackets with CUDA events (the roofline kernel); the
    # other launches run unbracketed there, and their times come from an
    # eager pass of the same steps after the timed region
    S.sense_profile_enable(True)
    for it in range(args.warmup):
        pipe.step(queries[it % nq], gate_sets[it % n_sets])
    torch.cuda.synchronize()
    warm = {name: S.sense_profile_query(name) for name in S.sense_profile_names()}
    live_family = max(warm, key=lambda name: warm[name][0])
    S.sense_profile_enable(False)
    if S.sense_device_status(clear=True) != 0:
        raise RuntimeError("device status bits set after warm-up")
    graph, graph_error = None, None
    if args.graph:
        try:
            graph = GraphStep(pipe, queries[0], gate_sets)
        except Exception as e:  # capture refused: time eager launches and say why
            graph_error = f"graph capture failed ({type(e).__name__}: {e}); eager launches timed"
            torch.cuda.synchronize()
    if graph is not None:
        for it in range(args.warmup):
            graph.step(queries[it % nq], it % n_sets)
        torch.cuda.synchronize()
        if S.sense_device_status(clear=True) != 0:
            raise RuntimeError("device status bits set after graph warm-up")

    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    graph_note = graph_error
    if graph is not None:
        # timed region: per step, copy the query into the staging buffer and
        # replay the captured step of this gate-input set
        e0.record(stream)
        for it in range(args.steps):
            graph.step(queries[it % nq], it % n_sets)
        e1.record(stream)
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        clk = clocks.stop()
        ms = e0.elapsed_time(e1)
        # CUDA events cannot time single kernels inside a replay: the
        # per-kernel times (roofline) come from an eager pass over the same
        # steps right after
        S.sense_profile_enable(True)
        for it in range(args.steps):
            pipe.step(queries[it % nq], gate_sets[it % n_sets])
        torch.cuda.synchronize()
        graph_note = (f"timed region: {args.steps} CUDA graph replays; kernel times from an "
                      f"eager pass of the same {args.steps} steps")
    else:
        S.sense_profile_enable(True)
        S.sense_profile_filter([live_family])
        e0.record(stream)
        for it in range(args.steps):
            pipe.step(queries[it % nq], gate_sets[it % n_sets])
        e1.record(stream)
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        clk = clocks.stop()
        ms = e0.elapsed_time(e1)
        live = S.sense_profile_query(live_family)
        # every family, from an eager pass of the same steps
        S.sense_profile_enable(True)
        for it in range(args.steps):
            pipe.step(queries[it % nq], gate_sets[it % n_sets])
        torch.cuda.synchronize()
        graph_note = (f"timed region: {args.steps} eager steps with CUDA events around the "
                      f"{live_family} launches only; the other kernels' times (kernel_ms) come "
                      f"from an eager pass of the same {args.steps} steps after it")
    prof = {name: S.sense_profile_query(name) for name in S.sense_profile_names()}
    if graph is None:
        prof[live_family] = live
    S.sense_profile_enable(False)
    ms = max_over_ranks(ms, dist, dev)
    launches = sum(v[1] for v in prof.values())

    # Supplementary: the same steps as CUDA graph replays (one graph per
    # gate-input set), after the eager timed region that the line reports.
    graph_line = None
    if graph is None and not args.no_graph_line:
        try:
            gstep = GraphStep(pipe, queries[0], gate_sets)
            for it in range(args.warmup):
                gstep.step(queries[it % nq], it % n_sets)
            torch.cuda.synchronize()
            if dist:
                dist.barrier()
            g0 = torch.cuda.Event(enable_timing=True)
            g1 = torch.cuda.Event(enable_timing=True)
            g0.record(stream)
            for it in range(args.steps):
                gstep.step(queries[it % nq], it % n_sets)
            g1.record(stream)
            torch.cuda.synchronize()
            gms = max_over_ranks(g0.elapsed_time(g1), dist, dev)
            if S.sense_device_status(clear=True) != 0:
                raise RuntimeError("device status bits set during graph replays")
            graph_line = {"value": job_throughput(cfg["q"] * args.steps, world, gms / 1e3),
                          "ms_per_step": gms / args.steps, "steps": args.steps,
                          "note": "the same steps replayed as one CUDA graph per gate-input "
                                  "set, timed after the eager region"}
            del gstep
        except Exception as e:  # capture refused: no supplementary line
            torch.cuda.synchronize()
            graph_line = {"value": None, "skipped": f"{type(e).__name__}: {e}"}

    q, n, d = cfg["q"], cfg["n"], cfg["d"]
    value = job_throughput(q * args.steps, world, ms / 1e3)
    peak, peak_kind = peaks()
    retrieval = {"kind": "exact"}
    if ann is None:
        # roofline of the dominant kernel (the key scan)
        scan_name = "scan_gemv" if q <= 8 else "scan_tc"
        scan_bytes_per_step = n * d * 2 + q * d * 2
        step_bytes = scan_bytes_per_step  # + the gate rows, added below
        per_row = NCU_TRAFFIC_PER_UNIT.get((scan_name, d))
        traffic = per_row * n if per_row else None
    else:
        # entries scanned per query (probed list sizes, over the distinct batches)
        off = ann["index"].arrays()["offsets"]
        sizes = off[1:] - off[:-1]
        scanned = []
        for b in range(min(nq, 64)):
            pipe.S.sense_project(queries[b], ann["basis"], ann["mean"], out=pipe.qproj)
            _, _, pr = S.sense_ivf_search(ann["index"], pipe.qproj, cfg["k"], ann["nprobe"],
                                          want_probes=True)
            scanned.append(sizes[pr.long()].sum(dim=1).float().mean().item())
        per_q = float(np.mean(scanned))
        v_, nl, pq_m = ann["v"], ann["nlist"], ann["pq_m"]
        entry = (pq_m if pq_m else 4 * v_) + 4 + 8  # payload + key index + pool write
        kb = {"project": v_ * d * 4 + q * d * 2 + q * v_ * 4,
              "ivf_coarse": nl * v_ * 4 + q * nl * 8,
              "ivf_scan": q * per_q * entry}
        if ann.get("rerank", 0):
            kb["rescore"] = q * ann["rerank"] * (d * 2 + 4)
        scan_name = max(kb, key=lambda name: prof.get(name, (0.0, 0))[0])
        scan_bytes_per_step = kb[scan_name]
        step_bytes = sum(kb.values())
        traffic = None
        # recall@k of the approximate top-k against (a) the exact top-k of the
        # full keys and (b) the exact top-k of the projected keys (a one-cell
        # flat index scans every projected key: the index's own loss)
        ex_ws = S.alloc_workspace(S.sense_retrieve_workspace_bytes(ds, q, cfg["k"]), dev)
        one = S.sense_ivf_build(ann["keys_proj"], ann["keys_proj"][:1].clone())
        hits, hits_p = [], []
        for b in range(min(nq, 64)):
            _, ex_i = S.sense_retrieve_topk(ds, queries[b], cfg["k"], workspace=ex_ws)
            pipe.retrieve(queries[b])
            # the one-call search keeps its projected query in its workspace
            S.sense_project(queries[b], ann["basis"], ann["mean"], out=pipe.qproj)
            _, px_i = S.sense_ivf_search(one, pipe.qproj, cfg["k"], 1)
            for a_row, e_row, p_row in zip(pipe.idx.cpu().tolist(), ex_i.cpu().tolist(),
                                           px_i.cpu().tolist()):
                hits.append(len(set(a_row) & set(e_row)) / len(e_row))
                hits_p.append(len(set(a_row) & set(p_row)) / len(p_row))
        del ex_ws, one
        ann.pop("keys_proj")
        retrieval = {"kind": ann["kind"], "proj_dim": v_, "nlist": nl, "nprobe": ann["nprobe"],
                     "pq_m": pq_m, "build_s": round(ann["build_s"], 3),
                     "pca_energy": ann["pca_energy"],
                     "mean_list": ann["mean_list"], "max_list": ann["max_list"],
                     "entries_scanned_per_query": per_q,
                     "rerank_candidates": ann.get("rerank", 0),
                     "recall_at_k_vs_exact": float(np.mean(hits)),
                     "recall_at_k_vs_exact_projected": float(np.mean(hits_p)),
                     "recall_queries": len(hits)}
    scan_ms, scan_launches = prof.get(scan_name, (0.0, 0))
    achieved = scan_bytes_per_step * args.steps / (scan_ms / 1e3) / 1e9 if scan_ms > 0 else 0.0

    # draft tree size (nodes per query) over a few steps, for draft tokens/s
    # and the loose trie's compression of the k*m candidate tokens (Sec. 4.3
    # "Loose Trie Compression"): distinct prefixes of the uncapped trie, on
    # the workload's spans and on spans that share prefixes within a key
    # cluster (the same retrieved indices)
    nodes, distinct, distinct_t, gate_rows_n = [], [], [], []
    tspans = synth.spans_cluster_template(assign, cfg["clusters"], cfg["m"], cfg["vocab"],
                                          seed=rank)
    tds = S.sense_datastore_build(keys, tspans)
    tdrafts = torch.empty_like(pipe.drafts)
    for it in range(16):
        pipe.step(queries[it % nq], gate_sets[it % n_sets])
        nodes.append(pipe.tree["num_nodes"].float().mean().item())
        # logits rows the gate must read: the root and every inner node
        par = pipe.tree["parent"].long()
        mark = torch.zeros(par.shape[0], par.shape[1] + 1, dtype=torch.int32, device=dev)
        mark.scatter_(1, par + 1, torch.ones_like(par, dtype=torch.int32))
        gate_rows_n.append(float(mark[:, 1:].sum().item() + par.shape[0]))
        full = S.sense_build_tree(pipe.drafts, node_cap=0)
        distinct.append(full["num_nodes"].float().mean().item())
        S.sense_gather_drafts(tds, pipe.idx, out=tdrafts)
        full = S.sense_build_tree(tdrafts, node_cap=0)
        distinct_t.append(full["num_nodes"].float().mean().item())
    del tds, tspans, tdrafts, full
    mean_nodes = float(np.mean(nodes))
    km = cfg["k"] * cfg["m"]

    # the gate's row pass dominates the sweep shapes: report whichever kernel
    # took longer, with its own algorithmic bytes
    gate_bytes_step = float(np.mean(gate_rows_n)) * cfg["vocab"] * 4
    step_bytes += gate_bytes_step
    g_ms, g_launches = prof.get("gate_rows", (0.0, 0))
    if g_ms > scan_ms:
        scan_name, scan_ms, scan_launches = "gate_rows", g_ms, g_launches
        scan_bytes_per_step = gate_bytes_step
        per_row = NCU_TRAFFIC_PER_UNIT.get(("gate_rows", cfg["vocab"]))
        traffic = per_row * float(np.mean(gate_rows_n)) if per_row else None
        achieved = scan_bytes_per_step * args.steps / (scan_ms / 1e3) / 1e9

    verify_info = None
    if args.verify:
        v = pipe.verify
        n_keys = v["prefix"] + v["L"]
        vbytes = 2 * v["heads"] * n_keys * 128 * 2 + v["heads"] * v["L"] * 128 * (2 + 4)
        vflops = 4 * v["heads"] * v["L"] * n_keys * 128
        t_ms, _ = prof.get("tree_attn", (0.0, 0))
        per = t_ms / args.steps / 1e3  # every attention launch of a step (main + any combine)
        verify_info = {"heads": v["heads"], "head_dim": 128, "draft_tokens": v["L"],
                       "prefix": v["prefix"], "cache_capacity": v["capacity"],
                       "us_per_step": per * 1e6,
                       "algorithmic_bytes": vbytes, "gbs": vbytes / per / 1e9 if per else None,
                       "frac_of_hbm": (vbytes / per / 1e9) / peak if per else None,
                       "tflops": vflops / per / 1e12 if per else None}

    def compression(dist):
        return {"distinct_prefixes": float(np.mean(dist)),
                "nodes_over_tokens": float(np.mean(dist)) / km,
                "compression": 1.0 - float(np.mean(dist)) / km}
    trie = {"candidate_tokens": km, "workload_spans": compression(distinct),
            "cluster_template_spans": compression(distinct_t),
            "capped_nodes": mean_nodes, "cap": pipe.cap}

    # end to end through the C ABI with host buffers
    e2e_steps = min(args.e2e_steps, args.steps)
    if gate_bytes > (1 << 30):
        e2e_steps = min(e2e_steps, 10)
    if gate_bytes > (4 << 30):
        e2e_steps = 0  # per-step inputs beyond host staging (reported as skipped)
    def packed(specs, device, pin):
        """One byte buffer holding tensors of the given (shape, dtype), each
        starting on a 256-byte boundary; returns the buffer and the views."""
        offs, total = [], 0
        for shape, dt in specs:
            offs.append(total)
            nbytes = int(np.prod(shape)) * torch.empty(0, dtype=dt).element_size()
            total += (nbytes + 255) // 256 * 256
        buf = torch.empty(total, dtype=torch.uint8, device=device)
        if pin:
            buf = buf.pin_memory()
        views = []
        for (shape, dt), off in zip(specs, offs):
            nbytes = int(np.prod(shape)) * torch.empty(0, dtype=dt).element_size()
            views.append(buf[off:off + nbytes].view(dt).view(shape))
        return buf, views

    h_query = torch.empty_like(queries[0], device="cpu").pin_memory()
    h_query.copy_(queries[0])
    d_query = torch.empty_like(queries[0])
    gsrc = gate_sets[0]
    # the gate's inputs travel as one pinned buffer and one copy
    gspecs = [(tuple(t.shape), t.dtype) for t in gsrc]
    if gate_bytes <= (4 << 30):
        h_gbuf, h_gate = packed(gspecs, "cpu", True)
        for hg, t in zip(h_gate, gsrc):
            hg.copy_(t)
        d_gbuf, d_gate = packed(gspecs, dev, False)
    else:
        h_gbuf = d_gbuf = None
        h_gate, d_gate = [], []
    # the step's results are written into one device buffer and read back
    # with one copy: the outputs of retrieval and of the gate are views of it
    ospecs = [((q, cfg["k"]), torch.float32), ((q, cfg["k"]), torch.int32),
              ((q, cfg["m"]), torch.int32)] + [((q,), torch.int32)] * 5 + \
             [((q, d), torch.bfloat16)]
    d_obuf, ov = packed(ospecs, dev, False)
    h_obuf = torch.empty_like(d_obuf, device="cpu").pin_memory()
    pipe.scores, pipe.idx = ov[0], ov[1]
    for name, t in zip(("accepted", "i_star", "L_star", "n_accept", "next_node", "next_anchor",
                        "h_next"), ov[2:]):
        pipe.gate[name] = t
    pipe.invalidate()
    h2d = h_query.numel() * h_query.element_size() + (h_gbuf.numel() if h_gbuf is not None else 0)
    d2h = h_obuf.numel()
    if e2e_steps == 0:
        h_gate = []
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    # the gate's inputs do not depend on retrieval: their host-to-device copy
    # runs on a side stream while the step drafts, and the gate waits for it
    copy_stream = torch.cuda.Stream(device=dev)
    copied = torch.cuda.Event()
    main = torch.cuda.current_stream()
    for it in range(e2e_steps):
        d_query.copy_(h_query, non_blocking=True)
        copy_stream.wait_stream(main)
        with torch.cuda.stream(copy_stream):
            if h_gate:
                d_gbuf.copy_(h_gbuf, non_blocking=True)
            copied.record(copy_stream)
        pipe.step(d_query, d_gate, before_gate=lambda: main.wait_event(copied))
        h_obuf.copy_(d_obuf, non_blocking=True)
        torch.cuda.current_stream().synchronize()
    e2e_s = max_over_ranks(time.perf_counter() - t0, dist, dev)
    e2e_value = job_throughput(q * e2e_steps, world, e2e_s) if e2e_steps else None

    base = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        if ann is None and not args.dynamic and not args.verify:
            base = cpu_baseline(cfg, keys, spans, queries, gate_sets)
        elif args.dynamic or args.verify:
            base = {"value": None, "skipped": "the oracle baseline times the static path only"}
        else:
            base = {"value": None, "skipped": "the oracle's index build over the full store "
                    "(fp32 loops in numpy) does not fit a bounded CPU sample"}

    if rank == 0:
        line = {
            "metric": METRIC,
            "value": value, "unit": "queries/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded clustered unit-norm keys, Zipf spans, N(0,9) logits)",
            "config": {"workload": args.workload, "retrieval": args.retrieval,
                       "keys": key_recipe,
                       "dynamic_capacity": args.dynamic, "verify_heads": args.verify,
                       **{k: cfg[k] for k in ("n", "d", "q", "k", "m", "vocab", "cap", "clusters")},
                       "key_bytes": n * d * 2,
                       "l2": f"inputs larger than L2: the {n * d * 2 / 1e9:.1f} GB store is "
                             "streamed every step",
                       "parallelism": f"replicas x{world}"},
            "retrieval": retrieval,
            "dynamic": dyn_info,
            "verify": verify_info,
            "launch": "cuda_graph" if graph is not None else "eager",
            "launch_note": graph_note,
            "graph_replay": graph_line,
            "hbm_gbs": step_bytes * args.steps / (ms / 1e3) / 1e9,
            "gate_rows_per_step": float(np.mean(gate_rows_n)),
            "draft_tokens_per_s": value * mean_nodes,
            # draft tokens (tree nodes) and raw gathered span tokens per second
            # of the drafting kernels alone (retrieval, gather, tree)
            "draft_tokens_per_s_drafting_kernels": draft_kernel_rate(prof, cfg["q"], mean_nodes,
                                                                     args.steps),
            "span_tokens_per_s_drafting_kernels": draft_kernel_rate(
                prof, cfg["q"], cfg["k"] * cfg["m"], args.steps),
            "mean_tree_nodes": mean_nodes,
            "trie_compression": trie,
            "roofline": {"bound": "hbm", "kernel": scan_name, "achieved": achieved,
                         "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                         "peak_kind": peak_kind,
                         "traffic": traffic,
                         "launches": scan_launches, "kernel_ms": scan_ms},
            "kernel_ms": {k: round(v[0], 4) for k, v in prof.items() if v[1]},
            "gpu_launches": launches,
            "clocks": clk,
            "e2e": ({"value": e2e_value, "unit": "queries/s", "h2d_bytes_per_step": h2d,
                     "d2h_bytes_per_step": d2h, "steps": e2e_steps} if e2e_steps else
                    {"value": None, "skipped": ("per-step gate inputs exceed 4 GB of host staging"
                                                if gate_bytes > (4 << 30) else "--e2e-steps 0")}),
            "cpu_baseline": base,
        }
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
