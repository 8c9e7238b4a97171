"""GB300-native scheduled denoiser step for spectral-guided static layer scheduling.

Modules: ``binding`` (ctypes binding of libsgd, the C ABI), ``schedule`` (offline
SCR/Frobenius scores and lifetimes), ``synth`` (seeded synthetic models/inputs),
``build`` (nvcc build of libsgd.so).  Importing the package loads nothing native;
``binding.lib()`` loads libsgd.so and raises if it is missing.
"""
