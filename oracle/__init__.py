"""Plain CPU oracle for the compressed-KV decode path (test infrastructure only).

This package is the slow, obviously-correct statement of what the GPU path
computes.  It is used ONLY by ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py``.  The product
library (``paper_2609_37988_gb300``) never imports it, and it imports nothing
from the product: the two share no code.  Inputs reach both sides from the
seeded generators in ``paper_2609_37988_gb300.workloads``, which hold none of
the method's arithmetic.

Modules
-------
quant      grouped asymmetric quantiser (fp32 op sequence), dequantisation
           (fp64), the paper's symmetric per-vector quantiser (Appendix C.3).
attention  layer -> source resolution (Sec. 2.1, depth axis), GQA decode and causal chunk (prefill) attention
           attention over dequantised caches, kept-position gather, MLA
           decode in the unabsorbed form (Appendix C.2).
evict      the attention-scored evictor composed with the cache (Sec. 3.4):
           votes summed over an observation window of queries, top
           positions per (sequence, KV head), kept lists.
cost       eq. (cost), eq. (compression), eq. (action space), eq. (range) and
           the metadata-inclusive storage accounting of Tab. realized_bits.
cache      whole-plan reference: builds every anchor's stored state from a
           per-layer plan (GQA anchors, and MLA anchors whose kept latent
           and positional key are stored as quantised vectors) and computes
           every layer's decode output.

Parity status: every function here is pinned by a ``-m "not gpu"`` test
(``tests/test_oracle_*.py``) against closed forms, the paper's printed
numbers, brute force, or a library routine.  No function is "parity unpinned".
"""
