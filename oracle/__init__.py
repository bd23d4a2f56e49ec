"""CPU oracle for the RateQuant packed mixed-bit KV path.

TEST INFRASTRUCTURE ONLY. Only the tests, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package. The product path (the C-ABI library and its Python binding) never
calls it and shares no code with it: no kernels, headers, helpers, tables or
pre/post-processing.

Everything here is plain, slow and written to be checked against the paper by
eye (RateQuant, arXiv 2605.06675):

* ``quant``     -- group-wise asymmetric min-max quantizer, its symmetric
                   absmax variant, and the randomized Hadamard pre-rotation
                   (Sec. 4.1 "Base quantizers", App. W "Quantizer
                   Implementation").
* ``pack``      -- the packed block format (codes + fp16 scale/zero); the paper
                   leaves storage unspecified, the format is this library's.
* ``calib``     -- distortion sweep D_i(b) and the log-linear fit of
                   D(b) = alpha * beta^-b (Assumption 1, Alg. 1 stage 2,
                   Sec. 3.4 "Distortion calibration", App. W "Outlier heads").
* ``alloc``     -- integer allocation: greedy max-heap (Alg. 1 stage 3,
                   Alg. 2, Prop. 3), exact DP for non-contiguous bit sets, and
                   continuous reverse waterfilling (Thm. 1 Eq. 2, App. B.1).
* ``attention`` -- decode attention on the dequantized cache, fp64.
* ``lloydmax``  -- Lloyd-Max codebook of N(0, 1) (Lloyd iteration + Newton)
                   and the RMS-normalised group quantizer that uses it
                   (App. F Table 8; TurboQuant's scalar quantizer, App. W).
* ``transfer``  -- cross-quantizer transfer matrix: allocate with one
                   quantizer's fitted model, score on another's measured
                   distortion (Sec. 3.4, Fig. 3; App. W Table 25).

Floating point: fp64 everywhere except the quantizer, whose steps are pinned
to fp32 / fp16 rounding (see ``quant``), because codes, scales and zero-points
are compared bit for bit.
"""
