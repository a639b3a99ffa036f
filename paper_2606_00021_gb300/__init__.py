"""Python binding of libsense: the SENSE drafting hot path on GB300.

Thin argument marshalling over the C ABI of include/sense.h: every function
here checks tensor devices, dtypes and shapes, allocates outputs with torch
when the caller did not pass them, and calls the function of the same name
in libsense.so on the current CUDA stream.  All computation happens in the
library's CUDA kernels; there is no CPU path.
"""
from __future__ import annotations

import contextlib
import ctypes as C
from dataclasses import dataclass, field

import torch

from . import _abi

SENSE_OK = 0
STATUS_NAMES = {0: "SENSE_OK", 1: "SENSE_ERR_INVALID_ARG", 2: "SENSE_ERR_UNSUPPORTED",
                3: "SENSE_ERR_OOM", 4: "SENSE_ERR_CUDA", 5: "SENSE_ERR_DEVICE_STATUS",
                6: "SENSE_ERR_TIMEOUT"}
DEVST_BAD_INDEX, DEVST_BAD_TOKEN, DEVST_TIMEOUT, DEVST_INTERNAL, DEVST_BAD_LENGTH = 1, 2, 4, 8, 16


class SenseError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


def lib():
    return _abi.load()


def _check(st: int):
    if st != SENSE_OK:
        msg = lib().sense_last_error().decode(errors="replace")
        raise SenseError(st, msg)


def _stream(stream) -> int:
    if stream is None:
        raw = getattr(torch._C, "_cuda_getCurrentRawStream", None)
        if raw is not None:
            return raw(torch.cuda.current_device())
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


class Prepared:
    """A library call whose arguments were marshalled once (device pointers,
    sizes, the stream).  Calling it issues the call again: the buffers keep
    their addresses and their contents may change between calls.  Returned by
    the prepare_* functions for per-step calls whose host-side marshalling
    would otherwise cost more than the kernels they launch."""

    def __init__(self, fn, args, keep):
        self._fn, self._args, self._keep = fn, args, keep

    def __call__(self):
        _check(self._fn(*self._args))


_recorder = None  # list of Prepared calls while record_calls() is active


def _call(fn, *args):
    """Runs a stream-ordered library call, or records it as a Prepared call
    inside record_calls()."""
    if _recorder is not None:
        _recorder.append(Prepared(fn, args, None))
        return
    _check(fn(*args))


@contextlib.contextmanager
def record_calls():
    """Inside the block the per-step library calls (retrieval, projection,
    search, re-scoring, gather, trie, masks, attention, dynamic buffer, gate)
    are recorded instead of run, with their arguments marshalled: the block
    yields the list of Prepared calls, to be issued again in order.  Output
    buffers the calls allocate are allocated once, here; every buffer must
    stay alive while the calls are used.  Calls that read results back to
    the host are not recorded and must not appear in the block."""
    global _recorder
    prev, _recorder = _recorder, []
    try:
        yield _recorder
    finally:
        _recorder = prev


def _ptr(t):
    return None if t is None else t.data_ptr()


def _need(t: torch.Tensor, name: str, dtype, ndim=None):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.device.type != "cuda":
        raise ValueError(f"{name} must be a CUDA tensor (got {t.device})")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype} (got {t.dtype})")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if ndim is not None and t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dims (got {tuple(t.shape)})")
    return t


def _i32(shape, dev):
    return torch.empty(shape, dtype=torch.int32, device=dev)


def sense_version() -> int:
    return int(lib().sense_version())


def sense_device_status(clear: bool = True, stream=None) -> int:
    """Status bits of the current device (synchronises the stream)."""
    out = C.c_uint32(0)
    st = lib().sense_device_status(C.c_void_p(_stream(stream)), C.byref(out), 1 if clear else 0)
    if st not in (0, 5, 6):
        _check(st)
    return int(out.value)


@dataclass
class Datastore:
    """Handle of a datastore (keys [n, d] bf16, spans [n, m] int32)."""
    handle: int
    n: int
    d: int
    m: int
    keys: torch.Tensor | None
    spans: torch.Tensor
    _keep: list = field(default_factory=list)

    def close(self):
        if self.handle:
            lib().sense_datastore_destroy(C.c_void_p(self.handle))
            self.handle = 0

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def sense_datastore_build(keys: torch.Tensor, spans: torch.Tensor, normalize: bool = False,
                          stream=None) -> Datastore:
    """Registers a datastore; keys bf16 [n, d] (borrowed) or f32 with normalize=True."""
    if normalize:
        _need(keys, "keys", torch.float32, 2)
        dtype_code, flags = 1, 1
    else:
        _need(keys, "keys", torch.bfloat16, 2)
        dtype_code, flags = 0, 0
    _need(spans, "spans", torch.int32, 2)
    n, d = keys.shape
    if spans.shape[0] != n:
        raise ValueError("keys and spans must have the same number of rows")
    out = C.c_void_p(0)
    _check(lib().sense_datastore_build(keys.data_ptr(), dtype_code, n, d, spans.data_ptr(),
                                       spans.shape[1], flags, C.c_void_p(_stream(stream)),
                                       C.byref(out)))
    ds = Datastore(out.value, n, d, spans.shape[1], keys if not normalize else None, spans)
    ds._keep = [keys, spans]
    return ds


class _DeviceArray:
    """Minimal __cuda_array_interface__ wrapper of a library-owned buffer."""

    def __init__(self, ptr: int, shape, typestr: str):
        self.__cuda_array_interface__ = {"shape": tuple(shape), "typestr": typestr,
                                         "data": (int(ptr), False), "version": 3,
                                         "strides": None}


def sense_datastore_keys(ds: Datastore) -> torch.Tensor:
    """The bf16 keys in use: the caller's tensor, or a zero-copy view of the
    normalised copy owned by the datastore (valid while ``ds`` is open)."""
    if ds.keys is not None:
        return ds.keys
    ptr = lib().sense_datastore_keys(C.c_void_p(ds.handle))
    view = torch.as_tensor(_DeviceArray(ptr, (ds.n, ds.d), "<i2"), device="cuda")
    return view.view(torch.bfloat16)


def sense_retrieve_workspace_bytes(ds: Datastore, q: int, k: int) -> int:
    return int(lib().sense_retrieve_workspace_bytes(C.c_void_p(ds.handle), q, k))


def alloc_workspace(nbytes: int, device=None) -> torch.Tensor:
    """Device scratch of at least nbytes, zero-filled (the soft gate keeps
    counters there that must start at zero)."""
    dev = device or torch.device("cuda", torch.cuda.current_device())
    return torch.zeros(max(int(nbytes), 256), dtype=torch.uint8, device=dev)


def sense_retrieve_topk(ds: Datastore, queries: torch.Tensor, k: int, out_scores=None,
                        out_idx=None, workspace=None, stream=None):
    """Exact top-k inner-product search: (scores f32 [q, k], idx int32 [q, k])."""
    _need(queries, "queries", torch.bfloat16, 2)
    q = queries.shape[0]
    if queries.shape[1] != ds.d:
        raise ValueError("queries must have d columns")
    dev = queries.device
    if out_scores is None:
        out_scores = torch.empty(q, k, dtype=torch.float32, device=dev)
    if out_idx is None:
        out_idx = _i32((q, k), dev)
    need = sense_retrieve_workspace_bytes(ds, q, k)
    if workspace is None:
        workspace = alloc_workspace(need, dev)
    _call(lib().sense_retrieve_topk, C.c_void_p(ds.handle), queries.data_ptr(), q, k,
          out_scores.data_ptr(), out_idx.data_ptr(),
          workspace.data_ptr(), workspace.numel(),
          C.c_void_p(_stream(stream)))
    return out_scores, out_idx


def sense_retrieve_topk_noalloc(ds: Datastore, queries: torch.Tensor, k: int, out_scores=None,
                                out_idx=None, stream=None):
    """Top-k search whose scratch is the library's fixed static device array.

    For callers that cannot allocate device memory or pass a workspace; the
    C entry point allocates nothing (only the outputs are allocated here when
    not given).  Requests larger than the static scratch raise SenseError."""
    _need(queries, "queries", torch.bfloat16, 2)
    q = queries.shape[0]
    if queries.shape[1] != ds.d:
        raise ValueError("queries must have d columns")
    dev = queries.device
    if out_scores is None:
        out_scores = torch.empty(q, k, dtype=torch.float32, device=dev)
    if out_idx is None:
        out_idx = _i32((q, k), dev)
    _check(lib().sense_retrieve_topk_noalloc(C.c_void_p(ds.handle), queries.data_ptr(), q, k,
                                             out_scores.data_ptr(), out_idx.data_ptr(),
                                             C.c_void_p(_stream(stream))))
    return out_scores, out_idx


def sense_retrieve_noalloc_status(clear: bool = True, stream=None) -> int:
    """Status bits the last allocation-free retrieval left (synchronises)."""
    out = C.c_uint32(0)
    st = lib().sense_retrieve_noalloc_status(C.c_void_p(_stream(stream)), C.byref(out),
                                             1 if clear else 0)
    if st not in (0, 5, 6):
        _check(st)
    return int(out.value)


def sense_retrieve_noalloc_selftest(limit_cycles: int = 200_000_000, stream=None) -> int:
    """Bounded-wait self test into the allocation-free retrieval's status
    word; returns the bits it left (SENSE_DEVST_TIMEOUT expected) without
    clearing them."""
    _check(lib().sense_retrieve_noalloc_selftest(C.c_void_p(_stream(stream)), int(limit_cycles)))
    return sense_retrieve_noalloc_status(clear=False, stream=stream)


def sense_rescore_topk(ds: Datastore, queries: torch.Tensor, cand_idx: torch.Tensor, k: int,
                       out_scores=None, out_idx=None, stream=None):
    """Exact scores of a shortlist of key indices per query (-1 = empty) and
    the top k of it by (score desc, index asc): Eq. 8's sim(h, k_i) over the
    approximate search's candidates."""
    _need(queries, "queries", torch.bfloat16, 2)
    _need(cand_idx, "cand_idx", torch.int32, 2)
    q, n_cand = cand_idx.shape
    if queries.shape != (q, ds.d):
        raise ValueError("queries must be [q, d] with q = cand_idx rows")
    dev = queries.device
    if out_scores is None:
        out_scores = torch.empty(q, k, dtype=torch.float32, device=dev)
    if out_idx is None:
        out_idx = _i32((q, k), dev)
    _call(lib().sense_rescore_topk, C.c_void_p(ds.handle), queries.data_ptr(), q,
          cand_idx.data_ptr(), n_cand, k, out_scores.data_ptr(),
          out_idx.data_ptr(), C.c_void_p(_stream(stream)))
    return out_scores, out_idx


def sense_gather_drafts(ds: Datastore, idx: torch.Tensor, anchor=None, n_keep=None,
                        force_anchor: bool = False, out=None, stream=None) -> torch.Tensor:
    """Candidate spans [q, n_keep, m] int32 for retrieved indices idx [q, k]."""
    _need(idx, "idx", torch.int32, 2)
    q, k = idx.shape
    keep = k if n_keep is None else int(n_keep)
    if anchor is not None:
        _need(anchor, "anchor", torch.int32, 1)
    if out is None:
        out = _i32((q, keep, ds.m), idx.device)
    _call(lib().sense_gather_drafts, C.c_void_p(ds.handle), idx.data_ptr(), q, k, _ptr(anchor),
          keep, 1 if force_anchor else 0, out.data_ptr(),
          C.c_void_p(_stream(stream)))
    return out


def sense_build_tree(spans: torch.Tensor, node_cap: int = 0, mask_bits: bool = False,
                     outs: dict | None = None, stream=None) -> dict:
    """Loose trie of spans [q, k, m]; returns a dict of device tensors."""
    _need(spans, "spans", torch.int32, 3)
    q, k, m = spans.shape
    cap = node_cap if node_cap > 0 else k * m
    dev = spans.device
    o = outs if outs is not None else {}
    o.setdefault("num_nodes", _i32((q,), dev))
    o.setdefault("tokens", _i32((q, cap), dev))
    o.setdefault("parent", _i32((q, cap), dev))
    o.setdefault("depth", _i32((q, cap), dev))
    o.setdefault("gamma", _i32((q, k, m), dev))
    if mask_bits:
        o.setdefault("mask_bits", torch.empty(q, cap, (cap + 31) // 32, dtype=torch.int32,
                                              device=dev))
    _call(lib().sense_build_tree, spans.data_ptr(), q, k, m, node_cap, 1 if mask_bits else 0,
          o["num_nodes"].data_ptr(), o["tokens"].data_ptr(),
          o["parent"].data_ptr(), o["depth"].data_ptr(),
          o["gamma"].data_ptr(), _ptr(o.get("mask_bits")),
          C.c_void_p(_stream(stream)))
    o["cap"] = cap
    return o


def sense_draft(ds: Datastore, queries: torch.Tensor, k: int, node_cap: int = 0,
                mask_bits: bool = False, outs: dict | None = None, workspace=None, stream=None,
                prepare: bool = False):
    """Retrieval, span gather and loose trie of one query batch in one call;
    the results of sense_retrieve_topk, sense_gather_drafts (no anchor) and
    sense_build_tree.  Returns a dict: scores, idx, spans and the tree
    arrays (num_nodes, tokens, parent, depth, gamma[, mask_bits], cap).
    With prepare=True nothing runs: returns (Prepared call, dict)."""
    _need(queries, "queries", torch.bfloat16, 2)
    q = queries.shape[0]
    if queries.shape[1] != ds.d:
        raise ValueError("queries must have d columns")
    m = ds.m
    cap = node_cap if node_cap > 0 else k * m
    dev = queries.device
    o = outs if outs is not None else {}
    o.setdefault("scores", torch.empty(q, k, dtype=torch.float32, device=dev))
    o.setdefault("idx", _i32((q, k), dev))
    o.setdefault("spans", _i32((q, k, m), dev))
    o.setdefault("num_nodes", _i32((q,), dev))
    o.setdefault("tokens", _i32((q, cap), dev))
    o.setdefault("parent", _i32((q, cap), dev))
    o.setdefault("depth", _i32((q, cap), dev))
    o.setdefault("gamma", _i32((q, k, m), dev))
    if mask_bits:
        o.setdefault("mask_bits", torch.empty(q, cap, (cap + 31) // 32, dtype=torch.int32,
                                              device=dev))
    if workspace is None:
        workspace = alloc_workspace(sense_retrieve_workspace_bytes(ds, q, k), dev)
    args = (C.c_void_p(ds.handle), queries.data_ptr(), q, k, workspace.data_ptr(),
            workspace.numel(), node_cap, 1 if mask_bits else 0, o["scores"].data_ptr(),
            o["idx"].data_ptr(), o["spans"].data_ptr(), o["num_nodes"].data_ptr(),
            o["tokens"].data_ptr(), o["parent"].data_ptr(), o["depth"].data_ptr(),
            o["gamma"].data_ptr(), _ptr(o.get("mask_bits")), C.c_void_p(_stream(stream)))
    o["cap"] = cap
    if prepare:
        return Prepared(lib().sense_draft, args, (ds, queries, workspace, dict(o))), o
    _call(lib().sense_draft, *args)
    return o


def sense_tree_mask_full(tree: dict, prefix_len: torch.Tensor, cache_len: int,
                         out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Additive static-KV attention mask [q, cap, cache_len] f32 of a tree
    built with mask_bits=True; prefix_len [q] int32 committed lengths."""
    bits = tree["mask_bits"]
    _need(bits, "mask_bits", torch.int32, 3)
    _need(tree["num_nodes"], "num_nodes", torch.int32, 1)
    _need(prefix_len, "prefix_len", torch.int32, 1)
    q, cap, _ = bits.shape
    if out is None:
        out = torch.empty(q, cap, cache_len, dtype=torch.float32, device=bits.device)
    _need(out, "out", torch.float32, 3)
    _call(lib().sense_tree_mask_full, bits.data_ptr(), tree["num_nodes"].data_ptr(), q, cap,
          prefix_len.data_ptr(), cache_len, out.data_ptr(),
          C.c_void_p(_stream(stream)))
    return out


# ---------------------------------------------------------------- approximate retrieval

def sense_project(x: torch.Tensor, basis: torch.Tensor, mean: torch.Tensor | None = None,
                  normalize: bool = True, out: torch.Tensor | None = None,
                  stream=None) -> torch.Tensor:
    """(x - mean) basis^T [n, v] f32 for bf16 rows x [n, d] (unit rows with
    ``normalize``): the query / key construction k = L2Norm(PCA(h))."""
    _need(x, "x", torch.bfloat16, 2)
    _need(basis, "basis", torch.float32, 2)
    n, d = x.shape
    v = basis.shape[0]
    if basis.shape[1] != d:
        raise ValueError("basis must be [v, d]")
    if mean is not None:
        _need(mean, "mean", torch.float32, 1)
    if out is None:
        out = torch.empty(n, v, dtype=torch.float32, device=x.device)
    _need(out, "out", torch.float32, 2)
    _call(lib().sense_project, x.data_ptr(), n, d, basis.data_ptr(), v, _ptr(mean),
          1 if normalize else 0, out.data_ptr(),
          C.c_void_p(_stream(stream)))
    return out


def sense_kmeans(x: torch.Tensor, init: torch.Tensor, iters: int, spherical: bool,
                 want_assign: bool = False, stream=None):
    """Lloyd's k-means on the rows of x [n, dim] f32 (rows may be strided, e.g.
    a column slice of a wider matrix) from seeds init [k, dim]; returns
    centroids (and the last round's assignment with ``want_assign``)."""
    if not isinstance(x, torch.Tensor) or x.dtype != torch.float32 or x.dim() != 2 \
            or x.device.type != "cuda" or x.stride(1) != 1:
        raise ValueError("x must be a CUDA float32 [n, dim] tensor with unit column stride")
    _need(init, "init", torch.float32, 2)
    n, dim = x.shape
    ld = x.stride(0) if n > 1 else dim
    k = init.shape[0]
    if init.shape[1] != dim:
        raise ValueError("init must be [k, dim]")
    cent = torch.empty(k, dim, dtype=torch.float32, device=x.device)
    assign = _i32((n,), x.device) if want_assign else None
    ws = alloc_workspace(lib().sense_kmeans_workspace_bytes(n, dim, k), x.device)
    _check(lib().sense_kmeans(x.data_ptr(), n, dim, ld, k, iters, 1 if spherical else 0,
                              init.data_ptr(), cent.data_ptr(), _ptr(assign), ws.data_ptr(),
                              ws.numel(), C.c_void_p(_stream(stream))))
    return (cent, assign) if want_assign else cent


def sense_ivf_residuals(vecs: torch.Tensor, centroids: torch.Tensor, stream=None):
    """(cell int32 [n], residual f32 [n, v]) of each vector."""
    _need(vecs, "vecs", torch.float32, 2)
    _need(centroids, "centroids", torch.float32, 2)
    n, v = vecs.shape
    cell = _i32((n,), vecs.device)
    res = torch.empty_like(vecs)
    _check(lib().sense_ivf_residuals(vecs.data_ptr(), n, v, centroids.data_ptr(),
                                     centroids.shape[0], cell.data_ptr(), res.data_ptr(),
                                     C.c_void_p(_stream(stream))))
    return cell, res


@dataclass
class IvfIndex:
    """Handle of an IVF-flat / IVF-PQ index (library-owned device memory)."""
    handle: int
    n: int
    v: int
    nlist: int
    pq_m: int
    max_list: int

    def close(self):
        if self.handle:
            lib().sense_ivf_destroy(C.c_void_p(self.handle))
            self.handle = 0

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def arrays(self) -> dict:
        """Zero-copy views of the lists (valid while the index is open)."""
        off, ids, pay = C.c_void_p(0), C.c_void_p(0), C.c_void_p(0)
        info = (C.c_int64 * 5)()
        _check(lib().sense_ivf_arrays(C.c_void_p(self.handle), info, C.byref(off), C.byref(ids),
                                      C.byref(pay)))
        view = lambda p, shape, ts: torch.as_tensor(_DeviceArray(p.value, shape, ts), device="cuda")
        out = {"offsets": view(off, (self.nlist + 1,), "<i8"), "ids": view(ids, (self.n,), "<i4")}
        if self.pq_m:
            out["codes"] = view(pay, (self.n, self.pq_m), "|u1")
        else:
            out["vectors"] = view(pay, (self.n, self.v), "<f4")
        return out


def sense_ivf_build(vecs: torch.Tensor, centroids: torch.Tensor,
                    codebooks: torch.Tensor | None = None, stream=None) -> IvfIndex:
    """IVF-flat (codebooks None) or IVF-PQ (codebooks [pq_m, 256, v/pq_m]) index."""
    _need(vecs, "vecs", torch.float32, 2)
    _need(centroids, "centroids", torch.float32, 2)
    n, v = vecs.shape
    pq_m = 0
    if codebooks is not None:
        _need(codebooks, "codebooks", torch.float32, 3)
        pq_m = codebooks.shape[0]
    out = C.c_void_p(0)
    _check(lib().sense_ivf_build(vecs.data_ptr(), n, v, centroids.data_ptr(), centroids.shape[0],
                                 _ptr(codebooks), pq_m, C.c_void_p(_stream(stream)),
                                 C.byref(out)))
    info = (C.c_int64 * 5)()
    _check(lib().sense_ivf_arrays(out, info, None, None, None))
    return IvfIndex(out.value, n, v, centroids.shape[0], pq_m, int(info[4]))


def sense_ivf_search_workspace_bytes(ix: IvfIndex, q: int, k: int, nprobe: int) -> int:
    return int(lib().sense_ivf_search_workspace_bytes(C.c_void_p(ix.handle), q, k, nprobe))


def sense_ann_draft(ix: "IvfIndex", ds: Datastore, queries: torch.Tensor, basis: torch.Tensor,
                    mean: torch.Tensor | None, k: int, nprobe: int, rerank: int = 0,
                    node_cap: int = 0, mask_bits: bool = False, outs: dict | None = None,
                    workspace=None, stream=None, prepare: bool = False):
    """Projection, IVF search (with optional exact re-scoring of `rerank`
    candidates), span gather and loose trie of one query batch in one call;
    the results of those calls one by one.  Returns a dict like sense_draft
    (with prepare=True: (Prepared call, dict), nothing run)."""
    _need(queries, "queries", torch.bfloat16, 2)
    _need(basis, "basis", torch.float32, 2)
    if mean is not None:
        _need(mean, "mean", torch.float32, 1)
    q = queries.shape[0]
    if queries.shape[1] != ds.d:
        raise ValueError("queries must have d columns")
    m = ds.m
    cap = node_cap if node_cap > 0 else k * m
    dev = queries.device
    o = outs if outs is not None else {}
    o.setdefault("scores", torch.empty(q, k, dtype=torch.float32, device=dev))
    o.setdefault("idx", _i32((q, k), dev))
    o.setdefault("spans", _i32((q, k, m), dev))
    o.setdefault("num_nodes", _i32((q,), dev))
    o.setdefault("tokens", _i32((q, cap), dev))
    o.setdefault("parent", _i32((q, cap), dev))
    o.setdefault("depth", _i32((q, cap), dev))
    o.setdefault("gamma", _i32((q, k, m), dev))
    if mask_bits:
        o.setdefault("mask_bits", torch.empty(q, cap, (cap + 31) // 32, dtype=torch.int32,
                                              device=dev))
    if workspace is None:
        need = lib().sense_ann_draft_workspace_bytes(C.c_void_p(ix.handle), q, k, nprobe, rerank)
        workspace = alloc_workspace(need, dev)
    args = (C.c_void_p(ix.handle), C.c_void_p(ds.handle), queries.data_ptr(), q,
            basis.data_ptr(), _ptr(mean), k, nprobe, rerank, node_cap, 1 if mask_bits else 0,
            workspace.data_ptr(), workspace.numel(), o["scores"].data_ptr(), o["idx"].data_ptr(),
            o["spans"].data_ptr(), o["num_nodes"].data_ptr(), o["tokens"].data_ptr(),
            o["parent"].data_ptr(), o["depth"].data_ptr(), o["gamma"].data_ptr(),
            _ptr(o.get("mask_bits")), C.c_void_p(_stream(stream)))
    o["cap"] = cap
    if prepare:
        return Prepared(lib().sense_ann_draft, args,
                        (ix, ds, queries, basis, mean, workspace, dict(o))), o
    _call(lib().sense_ann_draft, *args)
    return o


def sense_ann_search(ix: "IvfIndex", ds: Datastore, queries: torch.Tensor, basis: torch.Tensor,
                     mean: torch.Tensor | None, k: int, nprobe: int, rerank: int = 0,
                     out_scores=None, out_idx=None, workspace=None, stream=None):
    """sense_ann_draft's retrieval alone (projection, IVF search, optional
    exact re-scoring): (scores f32 [q, k], idx int32 [q, k])."""
    _need(queries, "queries", torch.bfloat16, 2)
    _need(basis, "basis", torch.float32, 2)
    if mean is not None:
        _need(mean, "mean", torch.float32, 1)
    q = queries.shape[0]
    if queries.shape[1] != ds.d:
        raise ValueError("queries must have d columns")
    dev = queries.device
    if out_scores is None:
        out_scores = torch.empty(q, k, dtype=torch.float32, device=dev)
    if out_idx is None:
        out_idx = _i32((q, k), dev)
    if workspace is None:
        need = lib().sense_ann_draft_workspace_bytes(C.c_void_p(ix.handle), q, k, nprobe, rerank)
        workspace = alloc_workspace(need, dev)
    _call(lib().sense_ann_search, C.c_void_p(ix.handle), C.c_void_p(ds.handle),
          queries.data_ptr(), q, basis.data_ptr(), _ptr(mean), k, nprobe, rerank,
          workspace.data_ptr(), workspace.numel(), out_scores.data_ptr(), out_idx.data_ptr(),
          C.c_void_p(_stream(stream)))
    return out_scores, out_idx


def sense_ivf_search(ix: IvfIndex, queries: torch.Tensor, k: int, nprobe: int,
                     out_scores=None, out_idx=None, want_probes: bool = False, workspace=None,
                     stream=None):
    """Approximate top-k: (scores f32 [q, k], idx int32 [q, k][, probes int32 [q, nprobe]])."""
    _need(queries, "queries", torch.float32, 2)
    q = queries.shape[0]
    if queries.shape[1] != ix.v:
        raise ValueError(f"queries must have {ix.v} columns")
    dev = queries.device
    if out_scores is None:
        out_scores = torch.empty(q, k, dtype=torch.float32, device=dev)
    if out_idx is None:
        out_idx = _i32((q, k), dev)
    probes = _i32((q, nprobe), dev) if want_probes else None
    if workspace is None:
        workspace = alloc_workspace(sense_ivf_search_workspace_bytes(ix, q, k, nprobe), dev)
    _call(lib().sense_ivf_search, C.c_void_p(ix.handle), queries.data_ptr(), q, k, nprobe,
          out_scores.data_ptr(), out_idx.data_ptr(), _ptr(probes),
          workspace.data_ptr(), workspace.numel(),
          C.c_void_p(_stream(stream)))
    return (out_scores, out_idx, probes) if want_probes else (out_scores, out_idx)


# ---------------------------------------------------------------- dynamic context buffer

@dataclass
class ContextBuffer:
    """Handle of a dynamic context buffer C_d (library-owned device ring)."""
    handle: int
    capacity: int
    d: int
    m: int

    def close(self):
        if self.handle:
            lib().sense_ctx_destroy(C.c_void_p(self.handle))
            self.handle = 0

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @property
    def count(self) -> int:
        """Positions appended so far (synchronises the current stream)."""
        out = C.c_int64(0)
        _check(lib().sense_ctx_count(C.c_void_p(self.handle), C.c_void_p(_stream(None)),
                                     C.byref(out)))
        return int(out.value)

    def reset(self, stream=None):
        _check(lib().sense_ctx_reset(C.c_void_p(self.handle), C.c_void_p(_stream(stream))))


def sense_ctx_create(capacity: int, d: int, m: int) -> ContextBuffer:
    out = C.c_void_p(0)
    _check(lib().sense_ctx_create(capacity, d, m, C.byref(out)))
    return ContextBuffer(out.value, capacity, d, m)


def sense_ctx_append(ctx: ContextBuffer, hidden: torch.Tensor, tokens: torch.Tensor, stream=None):
    """R.Update: hidden [t, d] bf16 states and the tokens [t] int32 they predicted."""
    _need(hidden, "hidden", torch.bfloat16, 2)
    _need(tokens, "tokens", torch.int32, 1)
    if hidden.shape[0] != tokens.shape[0] or hidden.shape[1] != ctx.d:
        raise ValueError("hidden must be [t, d] and tokens [t]")
    _call(lib().sense_ctx_append, C.c_void_p(ctx.handle), hidden.data_ptr(), tokens.data_ptr(),
          hidden.shape[0], C.c_void_p(_stream(stream)))


def sense_ctx_append_path(ctx: ContextBuffer, root_hidden: torch.Tensor,
                          node_hidden: torch.Tensor, gamma: torch.Tensor, i_star: torch.Tensor,
                          n_accept: torch.Tensor, accepted: torch.Tensor, stream=None):
    """R.Update of one verified step, on the device: root_hidden [d] and
    node_hidden [n_nodes, d] bf16, gamma [k, m], i_star / n_accept [1] and
    accepted [m] int32 (one query's tree and gate outputs)."""
    _need(root_hidden, "root_hidden", torch.bfloat16, 1)
    _need(node_hidden, "node_hidden", torch.bfloat16, 2)
    _need(gamma, "gamma", torch.int32, 2)
    for t, name in ((i_star, "i_star"), (n_accept, "n_accept"), (accepted, "accepted")):
        _need(t, name, torch.int32, 1)
    _call(lib().sense_ctx_append_path, C.c_void_p(ctx.handle), root_hidden.data_ptr(),
          node_hidden.data_ptr(), node_hidden.shape[0],
          gamma.data_ptr(), gamma.shape[0], i_star.data_ptr(),
          n_accept.data_ptr(), accepted.data_ptr(),
          C.c_void_p(_stream(stream)))


def sense_ctx_search(ctx: ContextBuffer, queries: torch.Tensor, k: int, delta: float = 0.0,
                     outs: dict | None = None, workspace=None, stream=None) -> dict:
    """DynSearch: dict of scores [q, k] (boosted), pos [q, k], spans [q, k, m]."""
    _need(queries, "queries", torch.bfloat16, 2)
    q = queries.shape[0]
    dev = queries.device
    o = outs if outs is not None else {}
    o.setdefault("scores", torch.empty(q, k, dtype=torch.float32, device=dev))
    o.setdefault("pos", torch.empty(q, k, dtype=torch.int64, device=dev))
    o.setdefault("spans", _i32((q, k, ctx.m), dev))
    if workspace is None:
        workspace = alloc_workspace(lib().sense_ctx_search_workspace_bytes(
            C.c_void_p(ctx.handle), q, k), dev)
    _call(lib().sense_ctx_search, C.c_void_p(ctx.handle), queries.data_ptr(), q, k,
          C.c_float(delta), o["scores"].data_ptr(), o["pos"].data_ptr(),
          o["spans"].data_ptr(), workspace.data_ptr(), workspace.numel(),
          C.c_void_p(_stream(stream)))
    return o


def sense_hybrid_drafts(ds: Datastore, static_scores: torch.Tensor, static_idx: torch.Tensor,
                        dyn: dict | None, anchor: torch.Tensor | None = None,
                        n_keep: int | None = None, force_anchor: bool = False, out=None,
                        stream=None) -> torch.Tensor:
    """Candidate drafts [q, n_keep, m] from static results and DynSearch results."""
    _need(static_scores, "static_scores", torch.float32, 2)
    _need(static_idx, "static_idx", torch.int32, 2)
    q, ks = static_idx.shape
    kd = 0 if dyn is None else dyn["scores"].shape[1]
    keep = ks + kd if n_keep is None else n_keep
    if anchor is not None:
        _need(anchor, "anchor", torch.int32, 1)
    if out is None:
        out = _i32((q, keep, ds.m), static_idx.device)
    _call(lib().sense_hybrid_drafts, C.c_void_p(ds.handle), static_scores.data_ptr(),
          static_idx.data_ptr(), ks,
          None if dyn is None else dyn["scores"].data_ptr(),
          None if dyn is None else dyn["spans"].data_ptr(), kd, q,
          _ptr(anchor), keep, 1 if force_anchor else 0,
          out.data_ptr(), C.c_void_p(_stream(stream)))
    return out


def sense_dyn_draft(ds: Datastore, ctx: ContextBuffer, queries: torch.Tensor,
                    static_scores: torch.Tensor, static_idx: torch.Tensor, kd: int,
                    delta: float = 0.0, anchor: torch.Tensor | None = None,
                    n_keep: int | None = None, force_anchor: bool = False, node_cap: int = 0,
                    mask_bits: bool = False, outs: dict | None = None, workspace=None,
                    stream=None) -> dict:
    """DynSearch, the hybrid rerank and the loose trie in one call: the dict
    of sense_ctx_search's outputs ("dyn": scores, pos, spans), the kept
    drafts ("spans" [q, n_keep, m]) and the tree (as sense_build_tree)."""
    _need(queries, "queries", torch.bfloat16, 2)
    _need(static_scores, "static_scores", torch.float32, 2)
    _need(static_idx, "static_idx", torch.int32, 2)
    if anchor is not None:
        _need(anchor, "anchor", torch.int32, 1)
    q, ks = static_idx.shape
    m = ctx.m
    keep = ks + kd if n_keep is None else n_keep
    cap = node_cap if node_cap > 0 else keep * m
    dev = queries.device
    o = outs if outs is not None else {}
    dyn = o.setdefault("dyn", {})
    dyn.setdefault("scores", torch.empty(q, kd, dtype=torch.float32, device=dev))
    dyn.setdefault("pos", torch.empty(q, kd, dtype=torch.int64, device=dev))
    dyn.setdefault("spans", _i32((q, kd, m), dev))
    o.setdefault("spans", _i32((q, keep, m), dev))
    o.setdefault("num_nodes", _i32((q,), dev))
    o.setdefault("tokens", _i32((q, cap), dev))
    o.setdefault("parent", _i32((q, cap), dev))
    o.setdefault("depth", _i32((q, cap), dev))
    o.setdefault("gamma", _i32((q, keep, m), dev))
    if mask_bits:
        o.setdefault("mask_bits", torch.empty(q, cap, (cap + 31) // 32, dtype=torch.int32,
                                              device=dev))
    if workspace is None:
        workspace = alloc_workspace(lib().sense_ctx_search_workspace_bytes(
            C.c_void_p(ctx.handle), q, kd), dev)
    _call(lib().sense_dyn_draft, C.c_void_p(ds.handle), C.c_void_p(ctx.handle),
          queries.data_ptr(), q, static_scores.data_ptr(), static_idx.data_ptr(), ks, kd,
          C.c_float(delta), _ptr(anchor), keep, 1 if force_anchor else 0, node_cap,
          1 if mask_bits else 0, workspace.data_ptr(), workspace.numel(),
          dyn["scores"].data_ptr(), dyn["pos"].data_ptr(), dyn["spans"].data_ptr(),
          o["spans"].data_ptr(), o["num_nodes"].data_ptr(), o["tokens"].data_ptr(),
          o["parent"].data_ptr(), o["depth"].data_ptr(), o["gamma"].data_ptr(),
          _ptr(o.get("mask_bits")), C.c_void_p(_stream(stream)))
    o["cap"] = cap
    return o


def sense_tree_attention(q: torch.Tensor, k_cache: torch.Tensor, vt_cache: torch.Tensor,
                         prefix_len: int, mask_bits: torch.Tensor, scale: float,
                         out: torch.Tensor | None = None, workspace=None,
                         stream=None) -> torch.Tensor:
    """Tree-masked attention of the verify forward: q [H, L, 128] bf16,
    k_cache [H, C, 128] and vt_cache [H, 128, C] bf16, mask_bits [>= L, words]
    int32 ancestor rows of one tree; returns out [H, L, 128] f32."""
    _need(q, "q", torch.bfloat16, 3)
    _need(k_cache, "k_cache", torch.bfloat16, 3)
    _need(vt_cache, "vt_cache", torch.bfloat16, 3)
    _need(mask_bits, "mask_bits", torch.int32, 2)
    heads, L, dh = q.shape
    cap = k_cache.shape[1]
    if out is None:
        out = torch.empty(heads, L, dh, dtype=torch.float32, device=q.device)
    if workspace is None:
        workspace = alloc_workspace(
            lib().sense_tree_attention_workspace_bytes(heads, L, prefix_len), q.device)
    _call(lib().sense_tree_attention, q.data_ptr(), k_cache.data_ptr(), vt_cache.data_ptr(), heads,
          L, dh, cap, prefix_len, mask_bits.data_ptr(),
          mask_bits.shape[1], C.c_float(scale), out.data_ptr(),
          workspace.data_ptr(), workspace.numel(),
          C.c_void_p(_stream(stream)))
    return out


def sense_soft_gate_workspace_bytes(q: int, cap: int, kappa: int) -> int:
    return int(lib().sense_soft_gate_workspace_bytes(q, cap, kappa))


def sense_soft_gate(tree: dict, root_logits: torch.Tensor, node_logits: torch.Tensor,
                    root_hidden: torch.Tensor, node_hidden: torch.Tensor, gamma: float = 0.05,
                    topk: int = 3, window: int = 6, tau: int = 0,
                    unnormalized_entropy: bool = False, want_G: bool = False,
                    workspace=None, outs: dict | None = None, stream=None,
                    prepare: bool = False):
    """Soft-gated evaluation of every draft path; returns a dict of device
    tensors (with prepare=True: (Prepared call, dict), nothing run)."""
    for name in ("num_nodes", "tokens", "parent", "gamma"):
        _need(tree[name], name, torch.int32)
    q, k, m = tree["gamma"].shape
    cap = tree["tokens"].shape[1]
    _need(root_logits, "root_logits", torch.float32, 2)
    _need(node_logits, "node_logits", torch.float32, 3)
    _need(root_hidden, "root_hidden", torch.bfloat16, 2)
    _need(node_hidden, "node_hidden", torch.bfloat16, 3)
    vocab = root_logits.shape[1]
    d = root_hidden.shape[1]
    if node_logits.shape != (q, cap, vocab) or node_hidden.shape != (q, cap, d):
        raise ValueError("node_logits / node_hidden must be [q, cap, V] / [q, cap, d]")
    dev = root_logits.device
    o = outs if outs is not None else {}
    for key in ("i_star", "L_star", "n_accept", "next_node", "next_anchor"):
        o.setdefault(key, _i32((q,), dev))
    o.setdefault("accepted", _i32((q, m), dev))
    o.setdefault("h_next", torch.empty(q, d, dtype=torch.bfloat16, device=dev))
    if want_G:
        o.setdefault("G", torch.empty(q, k, m, dtype=torch.uint8, device=dev))
    if workspace is None:
        workspace = alloc_workspace(sense_soft_gate_workspace_bytes(q, cap, topk), dev)
    p = _abi.GateParams(float(gamma), int(topk), int(window), int(tau),
                        1 if unnormalized_entropy else 0)
    args = (tree["tokens"].data_ptr(), tree["parent"].data_ptr(), tree["num_nodes"].data_ptr(),
            tree["gamma"].data_ptr(), q, k, m, cap, root_logits.data_ptr(),
            node_logits.data_ptr(), vocab, root_hidden.data_ptr(), node_hidden.data_ptr(), d,
            C.byref(p), o["i_star"].data_ptr(), o["L_star"].data_ptr(), o["n_accept"].data_ptr(),
            o["accepted"].data_ptr(), o["next_node"].data_ptr(), o["next_anchor"].data_ptr(),
            o["h_next"].data_ptr(), _ptr(o.get("G")), workspace.data_ptr(), workspace.numel(),
            C.c_void_p(_stream(stream)))
    if prepare:
        return Prepared(lib().sense_soft_gate, args,
                        (dict(tree), root_logits, node_logits, root_hidden, node_hidden, p,
                         workspace, dict(o))), o
    _call(lib().sense_soft_gate, *args)
    return o


def sense_selftest_timeout(limit_cycles: int = 200_000_000, stream=None) -> int:
    """Runs the bounded-wait self test and returns the device status bits
    it left (SENSE_DEVST_TIMEOUT expected); clears them afterwards."""
    _check(lib().sense_selftest_timeout(C.c_void_p(_stream(stream)), int(limit_cycles)))
    return sense_device_status(clear=True, stream=stream)


def sense_profile_enable(on: bool = True):
    _check(lib().sense_profile_enable(1 if on else 0))


def sense_profile_filter(names=None):
    """Bracket only these kernel families (iterable of names; None = all)
    while profiling is on; reset by sense_profile_enable."""
    arg = None if names is None else ",".join(names).encode()
    _check(lib().sense_profile_filter(arg))


def sense_profile_query(name: str):
    """(total device ms, launches) of one kernel family since profiling was enabled."""
    ms = C.c_double(0.0)
    n = C.c_int64(0)
    _check(lib().sense_profile_query(name.encode(), C.byref(ms), C.byref(n)))
    return float(ms.value), int(n.value)


def sense_profile_names():
    L = lib()
    return [L.sense_profile_name(i).decode() for i in range(L.sense_profile_count())]
