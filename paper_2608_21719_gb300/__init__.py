"""GB300-native paged GQA decode attention.

The compute path is the C-ABI library ``libps_decode.so`` (hand-written CUDA
for sm_103a); ``paper_2608_21719_gb300.ps_decode`` is its thin ctypes
binding.  Importing the binding fails loudly when the library has not been
built: there is no CPU fallback.

Submodules:
  ps_decode  -- binding to the C-ABI (argument marshalling only)
  inputs     -- seeded synthetic workloads (shared by the tests, the bench
                and the oracle's callers; no attention arithmetic)
  roofline   -- algorithmic byte accounting for the roofline figures
  build      -- nvcc build of the library
"""
