"""Oracle for skip-masked self-speculative decoding (KnapSpec, arXiv 2602.20217).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline leg may import anything here.  The CUDA path never
calls it, and it imports nothing from the CUDA path.

A plain, slow, fp64 numpy restatement of what the method computes:

* ``decoder``  - the target model as 2L sublayers (Sec. 2), the skip-masked
  draft f^(S), greedy parallel verification and acceptance (Sec. 2.1), the
  history of per-sublayer hidden states (Sec. 3.4).
* ``select``   - matrix cosine (Sec. 2), latency model (App. C), integer
  weight normalisation (Sec. 3.4), the 0/1 knapsack over sublayers with a
  brute-force checker (Sec. 3.3), expected tokens (Eq. 1), TPT (Eq. 3).

Each function is pinned by tests that do not re-type its formula; the pins are
listed in the tests' docstrings.
"""
