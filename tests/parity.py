"""Shared helpers of the parity tests: host copies and comparison rules.

Comparison rules (fixed before any kernel was written):
* scores: |gpu - oracle| <= 2e-3 absolute (fp32 accumulation of bf16
  products against an fp64 oracle on unit-norm keys);
* top-k indices: every index in one set but not the other has an oracle
  score within 2e-3 of the oracle's k-th score, and the order agrees except
  between entries whose oracle scores differ by less than 2e-3;
* spans, trees and gate decisions: bit-exact.
"""
import numpy as np
import torch

SCORE_TOL = 2e-3


def bits(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor -> uint16 bit patterns on the host."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def host(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().numpy()


def check_topk(gpu_scores, gpu_idx, oracle_scores_full, k, tol=SCORE_TOL):
    """Checks one query's GPU top-k against the oracle's full score row."""
    gs = np.asarray(gpu_scores, dtype=np.float64)
    gi = np.asarray(gpu_idx, dtype=np.int64)
    row = np.asarray(oracle_scores_full, dtype=np.float64)
    order = np.lexsort((np.arange(row.size), -row))
    oi = order[:k]
    t = row[oi[-1]]
    assert np.all(gi >= 0) and np.all(gi < row.size), "index out of range"
    assert len(set(gi.tolist())) == k, "duplicate indices"
    # scores of the returned keys match the oracle's scores of the same keys
    err = np.abs(gs - row[gi])
    assert err.max() <= tol, f"score error {err.max():.3g} > {tol}"
    diff = set(gi.tolist()) ^ set(oi.tolist())
    for i in diff:
        assert abs(row[i] - t) <= tol, f"index {i} (score {row[i]:.6f}) differs beyond tol from kth {t:.6f}"
    # order: non-increasing in oracle score up to tol
    os_ = row[gi]
    assert np.all(np.diff(os_) <= tol), "order disagrees beyond tolerance"
    return len(diff)
