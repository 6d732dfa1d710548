"""GB300-native Fast3Dcache cached denoising step.

``paper_2511_22533_gb300.f3dc`` is the thin ctypes binding of ``libf3dc.so``
(the C-ABI declared in ``include/f3dc.h``); ``synth`` holds the seeded
synthetic workload generators.  Importing the package does not load the CUDA
library; the binding loads it on first use and raises if it is missing.
"""
