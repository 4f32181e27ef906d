"""GB300-native FP8 token scoring with Calibrated Clipping.

The work runs in hand-written CUDA kernels for sm_103a behind the C ABI
declared in ``include/fp8rl.h`` (``libfp8rl.so``).  ``api`` is the thin Python
binding (argument marshalling over torch-owned device memory); ``synth`` draws
the seeded synthetic workloads.  Importing this package does not load the
native library; importing ``api`` does, and fails loudly if it is missing.
"""

__all__ = ["api", "synth"]
