"""CPU float64 oracle for the PS-PPO LM-head update pass.

TEST INFRASTRUCTURE ONLY. This package is the plain, slow, obviously-correct
statement of what the CUDA path computes. Only the tests, the smoke check and
the benchmark's CPU arms (its cpu_baseline and --impl reference) may import it;
the product path never does.
It shares no code with the CUDA path (no kernels, headers, helpers, tables or
constants): it is written directly from the paper.

Modules, in the order of the update pass:
  philox    Philox4x64-10 counter-based generator (Salmon et al., SC'11).
  cutoffs   cutoff sampling H ~ xi and inverse-survival weights 1/xi_t
            (Section 3.2, Eq. truncated_update_Ghat; Algorithm 1, steps 10-11).
  pack      group-normalised advantages (Section 3.1, broadcast advantage) and
            ragged prefix packing (Algorithm 1, step 11: only t <= H).
  lmhead    LM-head log-probabilities, clipped surrogate (Eq. 1), loss and the
            closed-form head gradient (Appendix D) composed with the surrogate.
  pipeline  the whole update pass in that order, and exact widening of bf16 inputs.
  design    the cutoff design upstream of the update: score proxy (Appendix D),
            reward-uncertainty proxy u_t (Appendix E, top-k of Appendix I) with the
            binarisation of continuous rewards (Appendix G), the budgeted monotone
            design with its cap (Section 3.3, Appendix F), the Section 4 variants,
            and the integer masses the sampler takes.

Every function is pinned by the tests in tests/test_oracle_*.py against facts
fixed by the paper or by mathematics (finite differences, exact enumeration of
the cutoff expectation, closed forms, library routines, brute force).
"""
