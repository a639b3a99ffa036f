"""GPU-vs-oracle parity of the tree-masked attention of the verify forward
(tcgen05 kernel), through the C ABI.  Inputs are seeded; the tree and its
ancestor bits come from the oracle's loose trie; expected values only from
``oracle``.

Tolerance: probabilities are rounded to bf16 (relative error <= 2^-9)
before the product with V, every sum is fp32, so |out - ref| <= 2^-9 max|V|
plus fp32 rounding; the test allows 2^-8 max|V| + 1e-5.
"""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from tests.parity import bits, host

pytestmark = pytest.mark.gpu
cuda = pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")


@pytest.fixture(scope="module")
def S():
    import paper_2606_00021_gb300 as S
    S.lib()
    return S


def _tree(seed, k, m_span, vocab, cap):
    rng = np.random.default_rng(seed)
    base = rng.integers(0, vocab, size=(max(1, k // 3), m_span))
    rows = base[rng.integers(0, base.shape[0], size=k)].copy()
    for r in range(k):
        cut = int(rng.integers(0, m_span + 1))
        rows[r, cut:] = rng.integers(0, vocab, size=m_span - cut)
    return O.loose_trie(rows[None], node_cap=cap, mask_bits=True)


@cuda
@pytest.mark.parametrize("heads,k,m_span,cap,prefix,capacity", [
    (2, 3, 3, 8, 5, 128), (4, 16, 8, 64, 300, 512), (32, 32, 16, 128, 3968, 4096),
    (3, 1, 1, 1, 0, 128), (8, 24, 8, 100, 1000, 1152), (1, 40, 16, 128, 130, 384),
    (4, 32, 16, 64, 2000, 2176),   # exactly 64 draft tokens (two lane quarters)
    (4, 32, 16, 65, 2000, 2176),   # one row into the third quarter
    # trees of <= 64 nodes (transposed products over 128-key blocks):
    (2, 16, 8, 64, 3000, 3200),    # 24 key splits: merged through the workspace
    (1, 8, 4, 32, 8000, 8192),     # 63 key splits (more than one warp of splits)
    (8, 24, 8, 64, 1000, 1152),    # tree keys straddle two key blocks; 9 splits
    (32, 24, 8, 64, 1000, 1152),   # the same in a cluster of 4 splits, one without blocks
    (4, 5, 4, 20, 0, 128),         # no committed prefix: every key is a tree node
    (6, 2, 16, 17, 129, 256),      # a 16-node chain and a branch, prefix past a block edge
])
def test_tree_attention_matches_oracle(S, heads, k, m_span, cap, prefix, capacity):
    dev = torch.device("cuda")
    tr = _tree(heads * 7 + k, k, m_span, 3, cap)
    L = int(tr["num_nodes"][0])
    assert 1 <= L <= 128 and prefix + L <= capacity
    D = 128
    q = synth.gaussian_rows_f32(heads * L, D, seed=1).reshape(heads, L, D).to(torch.bfloat16)
    kc = synth.gaussian_rows_f32(heads * capacity, D, seed=2).reshape(heads, capacity, D)
    vc = synth.gaussian_rows_f32(heads * capacity, D, seed=3).reshape(heads, capacity, D)
    kc, vc = kc.to(torch.bfloat16), vc.to(torch.bfloat16)
    mask = torch.from_numpy(tr["mask_bits"][0].view(np.int32)).to(dev)
    scale = 1.0 / np.sqrt(D)
    got = S.sense_tree_attention(q.to(dev), kc.to(dev), vc.transpose(1, 2).contiguous().to(dev),
                                 prefix, mask, scale)
    torch.cuda.synchronize()
    assert S.sense_device_status(clear=True) == 0
    M = O.mask_from_bits(tr["mask_bits"][0], L)
    want = O.tree_attention(bits(q), bits(kc), bits(vc), prefix, M, scale)
    vmax = np.abs(O.bf16_bits_to_f64(bits(vc[:, :prefix + L]))).max()
    err = np.abs(host(got).astype(np.float64) - want)
    assert err.max() <= 2.0 ** -8 * vmax + 1e-5, f"max error {err.max():.3g}"


@cuda
@pytest.mark.parametrize("heads,capacity,prefix", [(2, 1024, 900), (40, 4096, 3900)])
def test_tree_attention_large_logits_rescale(S, heads, capacity, prefix):
    """Keys aligned with the queries make later blocks' logits exceed the
    running maximum by far more than 2^8: the lazy rescale of O must keep the
    result exact within the tolerance (one key block per split, and about
    eleven blocks per split)."""
    dev = torch.device("cuda")
    tr = _tree(5, 8, 4, 3, 32)
    L = int(tr["num_nodes"][0])
    D = 128
    g = torch.Generator().manual_seed(4)
    q = torch.randn(heads, L, D, generator=g)
    kc = 0.05 * torch.randn(heads, capacity, D, generator=g)
    # growing alignment with the queries along the cache
    ramp = torch.linspace(0, 3, capacity)[None, :, None]
    kc = kc + ramp * q.mean(dim=1, keepdim=True) / q.mean(dim=1, keepdim=True).norm() * 4
    vc = torch.randn(heads, capacity, D, generator=g)
    q, kc, vc = q.to(torch.bfloat16), kc.to(torch.bfloat16), vc.to(torch.bfloat16)
    mask = torch.from_numpy(tr["mask_bits"][0].view(np.int32)).to(dev)
    got = S.sense_tree_attention(q.to(dev), kc.to(dev), vc.transpose(1, 2).contiguous().to(dev),
                                 prefix, mask, 1.0)
    torch.cuda.synchronize()
    assert S.sense_device_status(clear=True) == 0
    want = O.tree_attention(bits(q), bits(kc), bits(vc), prefix,
                            O.mask_from_bits(tr["mask_bits"][0], L), 1.0)
    vmax = np.abs(O.bf16_bits_to_f64(bits(vc[:, :prefix + L]))).max()
    err = np.abs(host(got).astype(np.float64) - want)
    assert np.isfinite(host(got)).all()
    assert err.max() <= 2.0 ** -8 * vmax + 1e-5, f"max error {err.max():.3g}"
