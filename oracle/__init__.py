"""CPU oracle for the WbG128 weight-only quantized linear layer (LAQuant, arXiv 2605.08755).

TEST INFRASTRUCTURE ONLY: the tests, the package's ``smoke()`` check and the benchmark's CPU
baseline leg may import this package; the product path never does.  It shares no code with the
CUDA library.

* ``oracle.c_oracle`` -- ctypes front end of ``laq_oracle.c`` (plain C, fp64): Eq. (1) RTN group
  quantizer, dequantizer, bit packing, and Y = X * W_hat.
* ``oracle.ref_numpy`` -- an independent numpy (float64) restatement of the same definitions,
  used to cross-check the C oracle bit for bit.
* ``oracle.decoder`` -- the operations of one decode step around the projections (RMSNorm,
  rotary embedding, grouped-query attention, SiLU * up, embedding, argmax) and the step itself.
* ``oracle.rotation`` -- the online pairwise rotation (channel scales, then rounds of Givens
  rotations per 128-channel group) that rotation-based methods run before each projection.
"""
