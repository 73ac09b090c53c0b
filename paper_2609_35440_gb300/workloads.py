"""The synthetic workloads the library is tested and measured on.

Shapes follow the readout sizes of the paper's pretraining models (Table
"Training FLOPs per token": d = 1024, 2048, 2560 at a 32k vocabulary, context
2048) and its use of synthetic Zipf-distributed tokens for systems runs
(Appendix on pipeline-parallel comparison, setup paragraph).  N is tokens per
module (micro-batch x 2048).  The vocabulary sweep uses V = 32000, 50304 and
128256.  No dataset item is reproduced: every tensor is drawn by ``synth``.
"""
from __future__ import annotations

from dataclasses import dataclass, replace


@dataclass(frozen=True)
class Workload:
    name: str
    K: int                 # modules sharing one readout
    N: int                 # tokens per module
    d: int                 # model width
    V: int                 # vocabulary size
    seed: int
    row_scale: bool = False        # per-row hidden scale, log-uniform in [0.5, 8]
    heavy_frac: float = 0.0        # fraction of W rows scaled x20
    targets: str = "uniform"       # "uniform" | "zipf"
    zipf_s: float = 1.1
    mask_frac: float = 0.0         # exact fraction of tokens set to ignore_index
    eps: float = 1e-6
    ignore_index: int = -100

    @property
    def M(self) -> int:
        return self.K * self.N

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


SMOKE = Workload("k2_n256_d128_v4096", K=2, N=256, d=128, V=4096, seed=0)
W340M = Workload("k4_n4096_d1024_v32000_zipf", K=4, N=4096, d=1024, V=32000,
                 seed=1, targets="zipf")
W1P3B = Workload("k4_n8192_d2048_v32000_rowscale_zipf_mask10", K=4, N=8192,
                 d=2048, V=32000, seed=2, row_scale=True, targets="zipf",
                 mask_frac=0.10)
W2B = Workload("k8_n16384_d2560_v32000_rowscale_zipf_mask10", K=8, N=16384,
               d=2560, V=32000, seed=3, row_scale=True, targets="zipf",
               mask_frac=0.10)


def vocab_sweep(V: int) -> Workload:
    return Workload(f"k4_n8192_d2048_v{V}_heavy_mask5", K=4, N=8192, d=2048,
                    V=V, seed=4, heavy_frac=0.01, targets="uniform",
                    mask_frac=0.05)


SWEEP = [vocab_sweep(V) for V in (32000, 50304, 128256)]

ALL = [SMOKE, W340M, W1P3B, W2B, *SWEEP]
BY_NAME = {w.name: w for w in ALL}

# The headline measurement: width 2048, vocabulary 32000, four modules.
HEADLINE = W1P3B
