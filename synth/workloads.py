"""Shapes of the synthetic workloads (the paper's model hidden sizes).

n keys of dimension d (bf16), q queries per batch, top-k, spans of m tokens
over a vocabulary, tree node cap (0 = uncapped), key clusters, span token
distribution, and the number of distinct query batches a benchmark cycles
through.
"""

WORKLOADS = {
    # tiny reference case: 4096 keys, all queries at once
    "tiny_4k": dict(n=4096, d=4096, q=8, k=8, m=8, vocab=32000, cap=64, clusters=64,
                    zipf=False, distinct=8),
    # LLaMA-7B hidden size, one query per decode step
    "llama7b_1m": dict(n=1048576, d=4096, q=1, k=32, m=16, vocab=32000, cap=64,
                       clusters=1024, zipf=True, distinct=512),
    # Qwen-7B hidden size, 16 sequences served together
    "qwen7b_4m": dict(n=4194304, d=3584, q=16, k=64, m=16, vocab=152064, cap=128,
                      clusters=4096, zipf=True, distinct=64),
    # LLaMA-70B hidden size, a 137 GB store
    "llama70b_8m": dict(n=8388608, d=8192, q=1, k=64, m=16, vocab=128256, cap=64,
                        clusters=8192, zipf=True, distinct=16),
    # retrieval + soft-gate sweep over k
    "sweep_2m_k16": dict(n=2097152, d=4096, q=64, k=16, m=16, vocab=128256, cap=0,
                         clusters=2048, zipf=True, distinct=64),
    "sweep_2m_k64": dict(n=2097152, d=4096, q=64, k=64, m=16, vocab=128256, cap=0,
                         clusters=2048, zipf=True, distinct=64),
    "sweep_2m_k256": dict(n=2097152, d=4096, q=64, k=256, m=16, vocab=128256, cap=0,
                          clusters=2048, zipf=True, distinct=64),
}
