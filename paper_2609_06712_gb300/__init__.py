"""RoLA hybrid attention for one GB300 (sm_103a).

The compute lives in hand-written CUDA kernels behind the C ABI of
``include/rola.h`` (``librola.so``, built by ``paper_2609_06712_gb300.build``).
``paper_2609_06712_gb300.rola`` is the thin Python binding with the same entry
points; importing it loads the library and fails loudly when it is missing.
"""
