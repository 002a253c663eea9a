"""CPU float64 oracle for the Truncated-BPTT meta-gradient (test infrastructure only).

This package is the correctness reference of the repository.  It is imported only by the
tests, by ``__graft_entry__.smoke()`` and by the CPU-baseline leg of ``bench.py``; the
library under ``paper_2505_00793_gb300`` never imports it and shares no code with it
(the only common module is the seeded input generator ``paper_2505_00793_gb300.synth``).

It computes exactly what Algorithm 1 of the paper (standard Truncated-BPTT, Section 2.3)
computes: the unrolled inner loop of Eq. 2 and ``dV/d eta`` through it by reverse-over-
reverse automatic differentiation (the inner gradient is itself recorded on the tape), with
per-inner-step checkpointing as in Section 4.  Arithmetic is plain PyTorch CPU ops in
float64; the only library "steps" are matmul, elementwise functions and torch.autograd.

Pins (``tests/test_oracle_pins.py``) tie it to things other than itself: central finite
differences of V(eta), the closed-form Hessian and meta-gradient of a linear model, the
symmetry u^T(Hv) = v^T(Hu), an explicit finite-difference Hessian, and special cases
(alpha = 0, T = 1, momentum 0).
"""
