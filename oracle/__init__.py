"""CPU oracle for Traversal Verification (arXiv 2505.12398).

TEST INFRASTRUCTURE ONLY. Nothing in the product path imports this package:
only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline / reference
legs of ``bench.py`` may use it.

The oracle is a plain, slow, literal restatement of the paper's algorithms in
float64 NumPy (or exact ``fractions.Fraction`` arithmetic for the pins):

* ``oracle.speculative`` -- single-token verification (Algorithm 1, §2.1) and
  Recursive Rejection Sampling with / without replacement (Algorithm 2, §2.2).
* ``oracle.traversal``   -- Traversal Verification (Algorithm 3, §3.1,
  Eqs. (1)-(3)), the per-tree state machine with materialised distributions.
* ``oracle.verify``      -- the boundary-shaped driver: logits, draft
  probabilities and pre-drawn uniforms in, accepted path / length / bonus out.
* ``oracle.exact``       -- exact enumeration of the output law (Lemma 1,
  Lemma 2, Theorems 1 and 2, Appendices A-B) used to pin the oracle.

It shares no code with the CUDA library under ``paper_2505_12398_gb300/``.
"""
