"""Plain fp64 CPU oracle for the frame-quantized linear layer (FrameQuant).

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg may
import this package.  The product library (libframequant and its Python binding) never imports
it and shares no code with it; the two meet only in the seeded input generators of workloads/.

  frames   tight fusion frame construction and random rotation (Sec. 2.2, Appendix J, K)
  quant    frame coefficients, 2-sigma clip, per-row RTN, de-noising gain (Sec. 3, Alg. 1, App. I)
  pack     the packed 2-bit code layout declared by the library header
  forward  analysis -> dequantized product -> synthesis (Sec. 3.2)
  layer    one call that builds a whole quantized layer from a workload
  gptq     the frame-domain GPTQ quantizer of Algorithm 1, step 4 (calibration Hessian)
  actquant rounding the frame representation of the activations to N-bit integers (App. F)

Parity status: every function is pinned by tests/test_oracle_*.py against brute force, closed
forms, printed examples or special cases; the de-noising gain (which the paper does not print) is
pinned as the empirical minimiser of the mean squared error under uniform rounding noise.
"""
