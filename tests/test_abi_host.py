"""Host-side checks of the C ABI: the library builds and loads without a GPU,
exports every function declared in include/sense.h, and rejects invalid
arguments before touching the device."""
import ctypes as C
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2606_00021_gb300 import _abi, _build
    _build.build()
    return _abi.load()


def _declared():
    src = open(os.path.join(ROOT, "include", "sense.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(sense_[a-z_0-9]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert len(names) >= 15
    for n in names:
        assert hasattr(lib, n), n
    from paper_2606_00021_gb300 import _abi
    assert set(names) == set(_abi.SIGNATURES), "binding and header disagree"


def test_every_declaration_cites_its_passage():
    """Each entry point of the header is documented by the comment before it
    (shared by a run of declarations): the paper's section, equation,
    algorithm or appendix it implements, or that the paper has none."""
    src = open(os.path.join(ROOT, "include", "sense.h")).read()
    decl = re.compile(r"\n(?:sense_status|size_t|const char\*|int32_t|int|void)\s+(sense_\w+)\s*\(")
    cite = re.compile(r"Sec\.|Eq\.|Alg\.|App\.|no\s+(?:\*\s+)?counterpart", re.S)
    found = 0
    for m in decl.finditer(src):
        before = src[:m.start()]
        end = before.rfind("*/")
        start = before.rfind("/*", 0, end)
        assert end > 0 and cite.search(before[start:end]), m.group(1)
        found += 1
    assert found >= 40


def test_status_strings(lib):
    assert lib.sense_status_string(0) == b"SENSE_OK"
    assert lib.sense_status_string(1) == b"SENSE_ERR_INVALID_ARG"
    assert lib.sense_status_string(6) == b"SENSE_ERR_TIMEOUT"
    assert lib.sense_version() >= 10000


def test_invalid_arguments_rejected_on_host(lib):
    p = C.c_void_p(16 * 1024)  # never dereferenced: validation fails first
    out = C.c_void_p(0)
    # datastore: bad n, d, m, alignment, flags
    assert lib.sense_datastore_build(p, 0, 0, 64, p, 4, 0, None, C.byref(out)) == 1
    assert lib.sense_datastore_build(p, 0, 10, 60, p, 4, 0, None, C.byref(out)) == 1
    assert lib.sense_datastore_build(p, 0, 10, 64, p, 33, 0, None, C.byref(out)) == 1
    assert lib.sense_datastore_build(C.c_void_p(16 * 1024 + 2), 0, 10, 64, p, 4, 0, None,
                                     C.byref(out)) == 1
    assert lib.sense_datastore_build(p, 0, 10, 64, p, 4, 0x80, None, C.byref(out)) == 1
    assert lib.sense_datastore_build(p, 0, 10, 64, p, 4, 1, None, C.byref(out)) == 1
    assert b"SENSE_DS_NORMALIZE" in lib.sense_last_error()
    # retrieve / gather on a NULL handle
    assert lib.sense_retrieve_topk(None, p, 1, 1, p, p, p, 1 << 20, None) == 1
    assert lib.sense_retrieve_topk_noalloc(None, p, 1, 1, p, p, None) == 1
    assert lib.sense_rescore_topk(None, p, 1, p, 8, 4, p, p, None) == 1
    assert lib.sense_draft(None, p, 1, 8, p, 1 << 20, 0, 0, p, p, p, p, p, p, p, p, None, None) == 1
    assert lib.sense_ann_draft(None, None, p, 1, p, None, 8, 4, 0, 0, 0, p, 1 << 20, p, p, p, p,
                               p, p, p, p, None, None) == 1
    assert lib.sense_ann_draft_workspace_bytes(None, 1, 8, 4, 0) == 0
    assert lib.sense_ann_search(None, None, p, 1, p, None, 8, 4, 0, p, 1 << 20, p, p, None) == 1
    assert lib.sense_dyn_draft(None, None, p, 1, p, p, 8, 4, 0.0, None, 8, 0, 0, 0, p, 1 << 20,
                               p, p, p, p, p, p, p, p, p, None, None) == 1
    # allocation-free status reader and self test: NULL output, limit range
    assert lib.sense_retrieve_noalloc_status(None, None, 1) == 1
    assert lib.sense_retrieve_noalloc_selftest(None, 0) == 1
    assert lib.sense_retrieve_noalloc_selftest(None, (1 << 34) + 1) == 1
    assert lib.sense_gather_drafts(None, p, 1, 1, None, 1, 0, p, None) == 1
    # tree: k, m, k*m, cap, flags
    args = (p, p, p, p, p, None, None)
    assert lib.sense_build_tree(p, 1, 0, 4, 0, 0, *args) == 1
    assert lib.sense_build_tree(p, 1, 4, 33, 0, 0, *args) == 1
    assert lib.sense_build_tree(p, 1, 1024, 16, 0, 0, *args) == 1
    assert lib.sense_build_tree(p, 1, 4, 4, -1, 0, *args) == 1
    assert lib.sense_build_tree(p, 1, 4, 4, 0, 1, *args) == 1  # mask bits without buffer
    # tree mask: q, cap, cache_len, NULL output
    assert lib.sense_tree_mask_full(p, p, 0, 8, p, 16, p, None) == 1
    assert lib.sense_tree_mask_full(p, p, 1, 0, p, 16, p, None) == 1
    assert lib.sense_tree_mask_full(p, p, 1, 8193, p, 16, p, None) == 1
    assert lib.sense_tree_mask_full(p, p, 1, 8, p, 0, p, None) == 1
    assert lib.sense_tree_mask_full(p, p, 1, 8, p, 16, None, None) == 1
    # gate parameters
    from paper_2606_00021_gb300._abi import GateParams
    gp = GateParams(0.05, 0, 6, 0, 0)
    ptrs = [p] * 4
    call = lambda g, v=128, d=64: lib.sense_soft_gate(*ptrs, 1, 4, 4, 16, p, p, v, p, p, d,
                                                      C.byref(g), *([p] * 7), None, p,
                                                      1 << 20, None)
    assert call(gp) == 1
    assert call(GateParams(0.05, 3, 0, 0, 0)) == 1
    assert call(GateParams(0.05, 3, 6, -1, 0)) == 1
    assert call(GateParams(0.05, 3, 6, 0, 0), v=130) == 1
    assert call(GateParams(0.05, 3, 6, 0, 0), d=60) == 1
    assert call(GateParams(float("nan"), 3, 6, 0, 0)) == 1


def test_extension_calls_reject_invalid_arguments(lib):
    p = C.c_void_p(16 * 1024)  # never dereferenced: validation fails first
    out = C.c_void_p(0)
    # projection: n, d, v, flags, alignment
    assert lib.sense_project(p, 0, 64, p, 16, None, 0, p, None) == 1
    assert lib.sense_project(p, 4, 60, p, 16, None, 0, p, None) == 1
    assert lib.sense_project(p, 4, 64, p, 129, None, 0, p, None) == 1
    assert lib.sense_project(p, 4, 64, p, 16, None, 0x10, p, None) == 1
    assert lib.sense_project(C.c_void_p(16 * 1024 + 4), 4, 64, p, 16, None, 0, p, None) == 1
    # k-means: dim, ld, k, workspace
    assert lib.sense_kmeans(p, 100, 12, 12, 8, 1, 0, p, p, None, p, 1 << 20, None) == 1
    assert lib.sense_kmeans(p, 100, 16, 8, 8, 1, 0, p, p, None, p, 1 << 20, None) == 1
    assert lib.sense_kmeans(p, 100, 16, 16, 0, 1, 0, p, p, None, p, 1 << 20, None) == 1
    assert lib.sense_kmeans(p, 100, 16, 16, 8, 1, 0, p, p, None, p, 16, None) == 1
    # IVF build: v, nlist, pq_m without codebooks, pq_m not dividing v
    assert lib.sense_ivf_build(p, 100, 24, p, 8, None, 0, None, C.byref(out)) == 1
    assert lib.sense_ivf_build(p, 100, 64, p, 20000, None, 0, None, C.byref(out)) == 1
    assert lib.sense_ivf_build(p, 100, 64, p, 8, None, 4, None, C.byref(out)) == 1
    assert lib.sense_ivf_build(p, 100, 64, p, 8, p, 3, None, C.byref(out)) == 1
    assert lib.sense_ivf_search(None, p, 1, 1, 1, p, p, None, p, 1 << 20, None) == 1
    # dynamic buffer: capacity below m, d not a multiple of 8
    assert lib.sense_ctx_create(4, 64, 8, C.byref(out)) == 1
    assert lib.sense_ctx_create(64, 60, 8, C.byref(out)) == 1
    assert lib.sense_ctx_search(None, p, 1, 1, C.c_float(0), p, p, p, p, 1 << 20, None) == 1
    assert lib.sense_hybrid_drafts(None, p, p, 4, p, p, 4, 1, None, 4, 0, p, None) == 1
    # tree attention: head dim, L, capacity, prefix beyond capacity, scale
    args = lambda hd, L, cap, pre, sc: (p, p, p, 2, L, hd, cap, pre, p, 4, C.c_float(sc), p, p,
                                        1 << 30, None)
    assert lib.sense_tree_attention(*args(64, 8, 128, 0, 0.1)) == 2
    assert lib.sense_tree_attention(*args(128, 129, 256, 0, 0.1)) == 1
    assert lib.sense_tree_attention(*args(128, 8, 100, 0, 0.1)) == 1
    assert lib.sense_tree_attention(*args(128, 8, 128, 125, 0.1)) == 1
    assert lib.sense_tree_attention(*args(128, 8, 128, 0, 0.0)) == 1
    # tree mask covered in test_invalid_arguments_rejected_on_host


def test_workspace_sizes(lib):
    assert lib.sense_retrieve_workspace_bytes(None, 1, 1) == 0
    assert lib.sense_soft_gate_workspace_bytes(2, 64, 3) >= 2 * 65 * 4
    assert lib.sense_soft_gate_workspace_bytes(2, 64, 3) % 256 == 0
