"""CPU oracle for TerMeZO (arxiv 2609.33548) -- TEST INFRASTRUCTURE ONLY.

A plain, slow, dense restatement of what the paper computes, written from
the paper in numpy (fp64 for continuous quantities; fp32 wherever the paper's
latents are stored or an fp32 value decides an integer code).  It shares no
code with the CUDA path and imports nothing from the package; only the test
suite, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` / reference arm
of ``bench.py`` may use it.  The product path never calls it.

Modules
  ternary  -- Eq. 2 quantizer, absmean scale, Eq. 3 boundary distance,
              2-bit packing of codes.
  philox   -- counter-based Philox-4x32-10 stream and Box-Muller normals
              (the perturbation z of Algorithm 1).
  bitnet   -- BitNet forward and minibatch loss (the minibatch objective of Eqs. 6-7).
  termezo  -- mask selection (Eqs. 4, 5), masked two-sided SPSA step
              (Eq. 1, Algorithm 1) and the boundary-crossing counters k_t, q_t of Eq. 11.

Parity status of each function is stated in its module header.
"""
