"""Seeded synthetic inputs for the TASP compiled sparse path.

This package is the input generator shared by the CPU oracle, the tests and
the benchmark. It holds no arithmetic of the method itself (no quantizer, no
mask construction, no forward pass): only a counter-based random generator,
an integer Irwin-Hall normal, FP32->BF16 rounding, and the keyed recipes that
say which seed, tensor id and index every synthetic value comes from.

The same generator is implemented a second time, independently, in CUDA inside
the library (for the multi-GB weight store and KV caches) and in C inside the
oracle (for fast regeneration of large layers); tests pin all three together.
"""
from .gen import *  # noqa: F401,F403
from .configs import *  # noqa: F401,F403
