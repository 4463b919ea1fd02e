"""CPU oracle for the masked MoE layer forward and the per-layer expert cache.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline /
reference legs of ``bench.py`` may import this package. The product path (the CUDA library and its
Python binding) never imports, links or executes anything here, and this package imports nothing from
the product path. The two share only the seeded input generator, which holds no step of the method.

Everything is a plain, slow, readable restatement of the paper's definitions in fp64 (numpy):

* ``routing``  - router logits, softmax, Top-K under a hard mask or a soft prior, gate weights
  (Section 3.1 Eq. topk; Section 3.2 Eq. stage1 and Eq. inference).
* ``ffn``      - SwiGLU expert, gated combine, shared experts (Section 3.1 Eq. topk).
* ``cache``    - per-layer expert cache with LRU / LFU / FIFO replacement, fetch accounting and the
  hit-rate / fetches-per-token metrics (Section 4.1 "Simulation", Eq. metrics), in two independent
  formulations.
* ``mask``     - Stage-1 mask sampling and the straight-through mask gradient (Section 3.2
  Eq. stage1 and Eq. ste).
* ``stack``    - the chained decode stack (residual stream, RMSNorm, one masked MoE block per layer)
  and the next-layer prediction that drives expert prefetch; the cache's prefetch event is in
  ``cache``.

Pins (tests marked ``not gpu``) tie each function to something other than itself; see the tests.
"""
from . import cache, ffn, mask, routing, stack  # noqa: F401
