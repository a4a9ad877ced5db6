"""Plain, slow CPU oracle for the P-PAS mixed-batch attention step.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path imports, calls or links
this package: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may use it.  It
shares no code with the CUDA path (no kernels, headers, helpers, tables or
pre/post-processing); the only thing both sides share is the seeded input
generator module, which holds none of the method's arithmetic.

Contents
--------
``oracle.attention``
    Paged causal GQA attention in float64 (the plain definition of scaled
    dot-product attention restricted to each query's causal prefix), written
    as un-page -> dense scores -> explicit mask -> max-subtracted softmax ->
    weighted sum of values.
``oracle.mlp``
    The gate-up projection of the decoder MLP profiled beside attention in
    Section 6.1: ``silu(X W_gate^T) * (X W_up^T)`` in float64.
``oracle.planner``
    The P-PAS step planner: Algorithm 1 (pressure test and prefill budget),
    chunked-prefill step composition under the unchanged global budget
    (Section 3), FIFO block allocation, block tables and slot mapping, and
    the request state update; plus the deterministic replay clock used for
    the burst-replay workload.

Every function cites the passage of the paper it follows.
"""
