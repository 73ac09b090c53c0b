"""fp64 CPU oracle of the SOLO shared-readout local loss.

Test infrastructure: only the tests, the smoke check and the CPU-baseline
leg of the benchmark import it.  It shares no code with the CUDA library.
All functions are pinned by tests against closed forms, invariants, finite
differences, brute force and an independent PyTorch fp64 composition.
"""
from .solo_oracle import *  # noqa: F401,F403
