"""CPU oracle for the Whisper-Flash speculative decode step (arxiv 2609.32869).

TEST INFRASTRUCTURE ONLY.  This package is a plain, slow, float64 numpy
restatement of what the paper's method computes; it exists to check the CUDA
path.  Only `tests/`, `__graft_entry__.smoke()` and the CPU-baseline leg of
`bench.py` may import it.  The product path never calls it, and it imports
nothing from the product package: the two share only the seeded input draws.

Modules
  philox     Philox4x32-10 counter-based generator (Salmon et al., SC'11) and
             the uniform / Gumbel draws made from it.
  decoder    Whisper-shaped target decoder, the Whisper-Flash drafter
             (Sec. 3.2, Eq. 2, App. A.2), prefill, plain greedy decoding
             (Eq. 1) and one speculative step (Sec. 3.1, App. A.1, A.4).
  acceptance greedy acceptance and the speculative rejection rule (Sec. 3.1).
"""
