"""FrameFT oracle: plain, slow, fp64 CPU reference of the adapter hot path.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports this package:
only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may use it.  It shares no code,
table or constant generator with the CUDA library; the two meet only on
seeded inputs produced by ``paper_2608_26430_gb300.workloads``.

Everything is written from the paper (FrameFT, arxiv 2608.26430):

* ``frames``  -- Spectral Tetris, modulation by k-th roots of unity,
  realification and Parseval normalisation (Sec. 3.2, Appendix "Example of
  fusion frames"), the dense synthesis matrix P and its structural pattern.
* ``support`` -- the random coefficient support shared across layers
  (Sec. 3.3) with a seeded splitmix64 stream.
* ``adapter`` -- dense C, the update dW = alpha/sqrt(mn) P_m C P_n^T
  (Sec. 3.1, Algorithm 1 steps 5-6), Y, dX, the coefficient gradient
  P_m^T grad_W P_n (Lemma 1 proof, Appendix A) and the multi-tenant merge.
* ``optim``   -- the AdamW step on the coefficient values and the linear
  learning-rate schedule with warmup (Appendix "Hyperparameters used for
  the experiments").

Parity status: every function is pinned by a ``-m "not gpu"`` test against
the printed worked example, closed forms (numpy FFT), invariants (tightness,
isometry, adjoint identities, linearity), finite differences, brute force,
or the library optimiser of PyTorch on the CPU (``optim``).
"""
