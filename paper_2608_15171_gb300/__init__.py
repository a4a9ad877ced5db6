"""GB300-native (sm_103a) mixed prefill+decode paged attention step behind P-PAS.

The compute path lives in the C-ABI shared library ``libppas.so`` built from
``csrc/`` (CUDA kernels for sm_103a plus a C++ host planner).
``paper_2608_15171_gb300.ppas`` is the thin ctypes binding with the same
names as the C entry points; importing it loads the library and fails loudly
when the library has not been built.  ``workloads`` holds the seeded input
generators.  Nothing is imported eagerly here.
"""
