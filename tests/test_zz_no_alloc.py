"""The allocation-free retrieval entry point agrees with the workspace one.

sense_retrieve_topk_noalloc serves callers that cannot allocate device
memory (their device memory is planned by another allocator, or their host
forbids cudaMalloc mid-request): it takes its scratch from a fixed static
device array instead of a caller workspace.  Its device-side checks report
into a status word inside that array, read by sense_retrieve_noalloc_status.
This file runs last so that a stop-at-first-failure run has already run
every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle as O
import synth
from tests.parity import bits, check_topk, host

pytestmark = pytest.mark.gpu


@pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")
def test_noalloc_matches_workspace_entry_point():
    import paper_2606_00021_gb300 as S
    dev = torch.device("cuda")
    n, d, k = 300001, 512, 32
    keys = synth.clustered_unit_keys(n, d, 256, seed=11, device=dev)
    spans = synth.spans_uniform(n, 4, 1000, seed=11, device=dev)
    ds = S.sense_datastore_build(keys, spans)
    full_cache = {}
    for call, (q, seed) in enumerate([(2, 5), (3, 6)]):  # two calls in a row
        qs, _ = synth.noisy_queries(keys, q, seed=seed)
        ref_s, ref_i = S.sense_retrieve_topk(ds, qs, k)
        got_s, got_i = S.sense_retrieve_topk_noalloc(ds, qs, k)
        torch.cuda.synchronize()
        assert torch.equal(got_i, ref_i), f"call {call}: indices differ"
        assert torch.equal(got_s, ref_s), f"call {call}: scores differ"
        full = O.scores(bits(keys), bits(qs))
        full_cache[call] = full
        for qi in range(q):
            check_topk(host(got_s[qi]), host(got_i[qi]), full[qi], k)


@pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")
def test_noalloc_rejects_oversize_request():
    import paper_2606_00021_gb300 as S
    dev = torch.device("cuda")
    n, d = 1 << 22, 8  # pool alone needs 8 queries x n x 8 bytes = 256 MiB
    keys = torch.zeros(n, d, dtype=torch.bfloat16, device=dev)
    spans = torch.zeros(n, 1, dtype=torch.int32, device=dev)
    ds = S.sense_datastore_build(keys, spans)
    qs = torch.zeros(8, d, dtype=torch.bfloat16, device=dev)
    with pytest.raises(S.SenseError) as e:
        S.sense_retrieve_topk_noalloc(ds, qs, 4)
    assert e.value.status == 2 and "static scratch" in str(e.value)


@pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")
def test_noalloc_alternates_paths_through_the_shared_array():
    """Consecutive calls that take the three retrieval paths (single pass
    for q <= 4, the sampled threshold for q <= 8, the tensor-core scan for
    q > 8) reuse the same static array; each must equal the workspace entry
    point bit for bit, whatever the previous call left in the array."""
    import paper_2606_00021_gb300 as S
    dev = torch.device("cuda")
    n, d = 100003, 512
    keys = synth.clustered_unit_keys(n, d, 128, seed=21, device=dev)
    spans = synth.spans_uniform(n, 4, 1000, seed=21, device=dev)
    ds = S.sense_datastore_build(keys, spans)
    kb = bits(keys)
    for call, (q, k, seed) in enumerate([(3, 32, 1), (8, 64, 2), (16, 64, 3), (3, 32, 4),
                                         (16, 200, 5), (1, 8, 6)]):
        assert S.sense_retrieve_workspace_bytes(ds, q, k) < (32 << 20) - 256
        qs, _ = synth.noisy_queries(keys, q, seed=seed)
        ref_s, ref_i = S.sense_retrieve_topk(ds, qs, k)
        got_s, got_i = S.sense_retrieve_topk_noalloc(ds, qs, k)
        torch.cuda.synchronize()
        assert S.sense_retrieve_noalloc_status(clear=True) == 0, f"call {call}: status bits"
        assert torch.equal(got_i, ref_i), f"call {call} (q={q}, k={k}): indices differ"
        assert torch.equal(got_s, ref_s), f"call {call} (q={q}, k={k}): scores differ"
        full = O.scores(kb, bits(qs))
        for qi in range(q):
            check_topk(host(got_s[qi]), host(got_i[qi]), full[qi], k)
    assert S.sense_device_status(clear=True) == 0


@pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")
def test_noalloc_status_word_reports_a_timed_out_wait():
    """A bounded wait that runs out (the self test waits on a barrier that
    nothing arrives on, then gives up) sets SENSE_DEVST_TIMEOUT in the
    allocation-free entry point's own status word; the reader returns it,
    clears it on request, and the device status word is not touched.  The
    next retrieval call starts from a clear word."""
    import paper_2606_00021_gb300 as S
    dev = torch.device("cuda")
    assert S.sense_retrieve_noalloc_status(clear=True) == 0
    bits_set = S.sense_retrieve_noalloc_selftest(limit_cycles=2_000_000)
    assert bits_set == 0x4  # SENSE_DEVST_TIMEOUT
    word = ctypes.c_uint32(0)
    st = S.lib().sense_retrieve_noalloc_status(ctypes.c_void_p(S._stream(None)),
                                               ctypes.byref(word), 0)
    assert st == 6 and word.value == 0x4  # SENSE_ERR_TIMEOUT, bit kept (clear = 0)
    assert S.sense_device_status(clear=False) == 0
    assert S.sense_retrieve_noalloc_status(clear=True) == 0x4
    assert S.sense_retrieve_noalloc_status(clear=True) == 0
    # set it again, then a retrieval call clears it before its own kernels
    assert S.sense_retrieve_noalloc_selftest(limit_cycles=2_000_000) == 0x4
    n, d, k = 5000, 256, 16
    keys = synth.clustered_unit_keys(n, d, 16, seed=31, device=dev)
    ds = S.sense_datastore_build(keys, synth.spans_uniform(n, 4, 100, seed=31, device=dev))
    qs, _ = synth.noisy_queries(keys, 2, seed=32)
    got_s, got_i = S.sense_retrieve_topk_noalloc(ds, qs, k)
    assert S.sense_retrieve_noalloc_status(clear=True) == 0
    ref_s, ref_i = S.sense_retrieve_topk(ds, qs, k)
    torch.cuda.synchronize()
    assert torch.equal(got_i, ref_i) and torch.equal(got_s, ref_s)
