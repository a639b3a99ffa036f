"""The allocation-free retrieval entry point agrees with the workspace one.

sense_retrieve_topk_noalloc serves callers that cannot allocate device
memory (their device memory is planned by another allocator, or their host
forbids cudaMalloc mid-request): it takes its scratch from a fixed static
device array instead of a caller workspace.  This file runs last so that a
stop-at-first-failure run has already run every other test.
"""
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
