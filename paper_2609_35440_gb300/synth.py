"""Seeded synthetic inputs shared by the CUDA path and the oracle.

This module holds no arithmetic of the method: it only draws the inputs
(hidden states, readout W, RMSNorm gain, targets) and quantises them to
bf16.  Both sides of every parity test take their inputs from here.

Random numbers come from a counter-based generator, SplitMix64 (Steele,
Lea, Flood, "Fast splittable pseudorandom number generators", OOPSLA 2014):
draw ``i`` of stream ``s`` under seed ``seed`` is
``mix(key(seed, s) + (i + 1) * 0x9E3779B97F4A7C15)``, so any slice of any
tensor can be regenerated on its own, in any order and on any machine.
Normals use the Box-Muller transform on consecutive pairs of uniforms.
Values are bit-identical wherever numpy's ``log``/``cos``/``sin`` agree to
the last bit; within one process both sides always see the same bytes.

Value recipe per workload (mirrors the paper's synthetic systems runs):

* hidden  h ~ N(0, 1), times a per-row scale log-uniform in [0.5, 8] when
  ``row_scale`` (stresses the RMSNorm);
* readout W ~ N(0, 0.02^2); exactly round(heavy_frac * V) distinct rows
  scaled x20 (heavy-tailed logits);
* gain gamma = 1 + N(0, 0.1^2);
* targets uniform in [0, V) or Zipf(s) with P(v) proportional to (v+1)^-s;
  exactly round(mask_frac * N) positions per module set to ignore_index.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from .workloads import Workload

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)

# stream ids
S_HIDDEN, S_ROWSCALE, S_W, S_HEAVY, S_GAMMA, S_TARGET, S_MASK = range(1, 8)

_CHUNK = 1 << 22


def _mix(z: np.ndarray) -> np.ndarray:
    z = (z ^ (z >> np.uint64(30))) * _M1
    z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def _key(seed: int, stream: int, sub: int = 0) -> np.uint64:
    with np.errstate(over="ignore"):
        k = np.array([seed], dtype=np.uint64)
        k = _mix(k + _GOLDEN)
        k = _mix(k ^ np.uint64(stream * 0x100000001B3 + sub))
    return k[0]


def raw_u64(seed: int, stream: int, start: int, count: int, sub: int = 0) -> np.ndarray:
    """Draws ``start .. start+count-1`` of one stream as uint64."""
    key = _key(seed, stream, sub)
    idx = np.arange(start + 1, start + count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return _mix(key + idx * _GOLDEN)


def uniform(seed, stream, start, count, sub=0) -> np.ndarray:
    """Uniform doubles in the open interval (0, 1)."""
    bits = raw_u64(seed, stream, start, count, sub) >> np.uint64(11)
    return (bits.astype(np.float64) + 0.5) * (1.0 / 9007199254740992.0)


def normal(seed, stream, start, count, sub=0) -> np.ndarray:
    """Standard normals; element i uses the uniform pair (2*(i//2), 2*(i//2)+1)."""
    p0 = start // 2
    p1 = (start + count + 1) // 2
    u = uniform(seed, stream, 2 * p0, 2 * (p1 - p0), sub).reshape(-1, 2)
    rad = np.sqrt(-2.0 * np.log(u[:, 0]))
    ang = 2.0 * np.pi * u[:, 1]
    pair = np.stack([rad * np.cos(ang), rad * np.sin(ang)], axis=1).reshape(-1)
    off = start - 2 * p0
    return pair[off:off + count]


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Quantises doubles to bf16 bit patterns (uint16) via float32, ties to even."""
    f = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounding = np.uint32(0x7FFF) + ((f >> np.uint32(16)) & np.uint32(1))
    return ((f + rounding) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32)


def _perm_prefix(seed, stream, n, m, sub) -> np.ndarray:
    """The first m positions of a seeded uniform random permutation of range(n)."""
    if m <= 0:
        return np.zeros(0, dtype=np.int64)
    u = uniform(seed, stream, 0, n, sub)
    return np.sort(np.argsort(u, kind="stable")[:m])


@dataclass
class Inputs:
    hidden: np.ndarray      # uint16 bf16 bits [K, N, d]
    W: np.ndarray           # uint16 bf16 bits [V, d]
    gamma: np.ndarray       # uint16 bf16 bits [d]
    targets: np.ndarray     # int32 [K, N]; ignore_index where masked
    mask: np.ndarray | None = None   # optional uint8 [K, N]; 0 = masked


def gen_hidden(wl: Workload, k: int, row0: int = 0, rows: int | None = None) -> np.ndarray:
    """bf16 bits of hidden rows [row0, row0+rows) of module k, shape [rows, d]."""
    rows = wl.N - row0 if rows is None else rows
    d = wl.d
    out = np.empty((rows, d), dtype=np.uint16)
    step = max(1, _CHUNK // d)
    for r in range(0, rows, step):
        nr = min(step, rows - r)
        start = (row0 + r) * d
        h = normal(wl.seed, S_HIDDEN, start, nr * d, sub=k).reshape(nr, d)
        if wl.row_scale:
            u = uniform(wl.seed, S_ROWSCALE, row0 + r, nr, sub=k)
            h = h * (0.5 * np.power(16.0, u))[:, None]
        out[r:r + nr] = to_bf16_bits(h)
    return out


def gen_W(wl: Workload) -> np.ndarray:
    V, d = wl.V, wl.d
    out = np.empty((V, d), dtype=np.uint16)
    heavy = np.zeros(V, dtype=bool)
    nh = int(round(wl.heavy_frac * V))
    heavy[_perm_prefix(wl.seed, S_HEAVY, V, nh, 0)] = True
    step = max(1, _CHUNK // d)
    for r in range(0, V, step):
        nr = min(step, V - r)
        w = 0.02 * normal(wl.seed, S_W, r * d, nr * d).reshape(nr, d)
        w[heavy[r:r + nr]] *= 20.0
        out[r:r + nr] = to_bf16_bits(w)
    return out


def gen_gamma(wl: Workload) -> np.ndarray:
    return to_bf16_bits(1.0 + 0.1 * normal(wl.seed, S_GAMMA, 0, wl.d))


def gen_targets(wl: Workload) -> np.ndarray:
    K, N, V = wl.K, wl.N, wl.V
    y = np.empty((K, N), dtype=np.int32)
    if wl.targets == "zipf":
        w = np.power(np.arange(1, V + 1, dtype=np.float64), -wl.zipf_s)
        cdf = np.cumsum(w)
        cdf /= cdf[-1]
    for k in range(K):
        u = uniform(wl.seed, S_TARGET, 0, N, sub=k)
        if wl.targets == "zipf":
            t = np.searchsorted(cdf, u, side="right")
        elif wl.targets == "uniform":
            t = np.floor(u * V)
        else:
            raise ValueError(wl.targets)
        y[k] = np.minimum(t, V - 1).astype(np.int32)
        nm = int(round(wl.mask_frac * N))
        y[k, _perm_prefix(wl.seed, S_MASK, N, nm, k)] = wl.ignore_index
    return y


def generate(wl: Workload) -> Inputs:
    hidden = np.stack([gen_hidden(wl, k) for k in range(wl.K)])
    return Inputs(hidden=hidden, W=gen_W(wl), gamma=gen_gamma(wl),
                  targets=gen_targets(wl))


def random_mask(seed: int, K: int, N: int, frac: float) -> np.ndarray:
    """A uint8 [K, N] keep-mask (0 = masked) with exactly round(frac*N) zeros per module."""
    m = np.ones((K, N), dtype=np.uint8)
    for k in range(K):
        m[k, _perm_prefix(seed, S_MASK, N, int(round(frac * N)), 1000 + k)] = 0
    return m


S_TAU, S_BIAS = 8, 9


def gen_heads(wl: Workload, tau_spread: float = 0.5, bias_std: float = 0.5):
    """Heads' parameters (fp32): temperatures tau_k = 1 + tau_spread * U(-1, 1) for
    the auxiliary modules and 1 for the terminal; biases b_k ~ N(0, bias_std^2)."""
    tau = (1.0 + tau_spread * (2.0 * uniform(wl.seed, S_TAU, 0, wl.K) - 1.0)).astype(np.float32)
    tau[-1] = 1.0
    bias = np.empty((wl.K, wl.V), dtype=np.float32)
    for k in range(wl.K):
        bias[k] = bias_std * normal(wl.seed, S_BIAS, 0, wl.V, sub=k)
    return tau, bias
