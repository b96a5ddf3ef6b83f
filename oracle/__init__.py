"""Plain, slow, fp64 CPU oracle for the ZO-Act per-step hot path.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The product (the CUDA library and its Python binding) never imports,
links or executes anything here, and nothing here imports the product.

Every function states the passage of the ZO-Act paper (arXiv 2607.01125) it
writes out:

* ``philox``  -- the Gaussian perturbation Z (Section 3, "ZO-Act": Z ~ N(0, I)),
  drawn from Philox4x32-10 (Salmon et al., SC'11) with Box-Muller.
* ``layers``  -- the adapted linear W_eff = W + V_r (B + mu Z) and its perturbed
  forward pass Y+ = XW + (X V_r)(B + mu Z)  (Section 3), the INT4 group
  dequantisation of the frozen weight, and the glue ops of the synthetic graphs.
* ``loss``    -- the loss pair and the projected-gradient scalar a (Section 3
  estimator; Algorithm 2), in the two-sided form.
* ``optim``   -- Adam on the estimated coefficient gradient (Section 3; Section 5
  setup; Appendix B tables: weight decay 0).
* ``basis``   -- Algorithm 1 (top-r right singular vectors of the calibration
  activations), a hand-written cyclic Jacobi eigensolver used as its pin, and
  the randomised subspace iteration that reaches the same subspace.
* ``graphs``  -- the synthetic model graphs that chain adapted linears.

Pinned: every function has at least one ``-m "not gpu"`` test in ``tests/``
against a value or property fixed by the paper or by mathematics (known-answer
vectors, closed forms, invariants, brute force, textbook special cases).
"""
