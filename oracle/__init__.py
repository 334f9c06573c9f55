"""CPU oracle for the CLEAR-MoE FFN forward (arxiv 2606.28516). TEST INFRASTRUCTURE ONLY.

A plain, slow, float64 restatement of the paper's inference layer, written from Eq. 2 and
Algorithm 3 ("CLEAR-MoE FFN Inference (Grouped backend)"), used to prove the CUDA library
right. Only the tests, the smoke check and the CPU-baseline leg of the benchmark may import it;
the library never calls it and shares no code with it.

Modules:
  clearmoe -- router, argmax routing, fc1 + GELU, shared basis, residual experts, dense FFN,
              the 12-sublayer stack (numpy float64; a matmul is the only library step)
  brute    -- pure-Python per-element loops on tiny shapes, used to pin `clearmoe`
  clearmoe_ref.c, ref_c
           -- the same layer in plain C (float64 loops, libm erf), loaded through ctypes; it
              shares no code with the other two and is checked against them and the golden
              values (tests/test_oracle_c.py)

Parity status: every function in `clearmoe` is pinned (tests/test_oracle_pins.py) against
closed forms, hand-derived golden values (tests/golden/), the brute force and the paper's
algebraic identities (dense reduction, the D3 full-residual identity, the scalar-residual form).
"""
