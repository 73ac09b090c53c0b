"""SOLO shared-readout local loss on one GB300 (sm_103a).

The compute lives in the C-ABI library ``libsolo_readout.so`` built from
``csrc/``; ``solo_readout`` is its thin ctypes binding.  Importing this
package does not load the library, so the seeded input generator
(``synth``) and the workload table (``workloads``) stay usable on a machine
without a GPU.
"""

__all__ = ["workloads", "synth"]
