"""CPU oracle for the SENSE drafting hot path (test infrastructure only).

Imported only by the tests, the smoke check and the CPU-baseline legs of the
benchmark; the product library never uses it.
"""
from .sense_oracle import (  # noqa: F401
    bf16_bits_to_f64,
    f64_to_bf16_bits,
    gather_drafts,
    loose_trie,
    loose_trie_alg3,
    mask_from_bits,
    normalize_keys_bf16,
    scores,
    soft_gate,
    topk,
    tree_attention,
    tree_mask_full,
)
