"""FLOP and byte accounting of the readout path (paper, Appendix H cost model).

Per token a block costs b = 12 d^2 + 2 T d multiply-accumulates, a full
vocabulary readout r = V d.  Counting one forward pass as one unit, the
terminal readout costs 3r (forward, input gradient, weight gradient) and an
auxiliary readout 2r (forward and input gradient only: its weights are a
detached copy).  One multiply-accumulate is two FLOPs.

For one call of the library over K modules of N tokens, the algorithmic
tensor work is therefore (2K + 1) * 2 N V d FLOPs.  The library executes
exactly that many: the backward pass reuses the forward's exponentials
instead of recomputing the logits.
"""
from __future__ import annotations


def block_macs(d: int, T: int) -> int:
    return 12 * d * d + 2 * T * d


def readout_macs(V: int, d: int) -> int:
    return V * d


def per_token_gflops(L: int, d: int, K: int, H: int, T: int, V: int) -> dict:
    """The columns of the paper's 'Training FLOPs per token' table, in GFLOP."""
    b, r = block_macs(d, T), readout_macs(V, d)
    layers = 3 * L * b * 2
    aux_blocks = 3 * (K - 1) * H * b * 2
    readouts = (2 * K + 1) * r * 2
    bp_total = layers + 3 * r * 2
    solo_total = layers + aux_blocks + readouts
    g = 1e-9
    return dict(bp_total=bp_total * g, bp_layers=layers * g,
                solo_total=solo_total * g, aux_blocks=aux_blocks * g,
                readouts=readouts * g, rho=solo_total / bp_total)


def rho(L: int, d: int, K: int, H: int, T: int, V: int) -> float:
    """Work ratio of Eq. 6: W_SOLO / W_BP."""
    gam = V / (L * (12 * d + 2 * T))
    return (1 + (K - 1) * H / L + (2 * K + 1) * gam / 3) / (1 + gam)


def readout_broadcast_bytes(p: int, V: int, d: int, elem_bytes: int = 2) -> int:
    """Bytes of one readout broadcast from the last of p stages: (p-1)(Vd+V) numbers."""
    return (p - 1) * (V * d + V) * elem_bytes


def call_flops(K: int, N: int, d: int, V: int) -> float:
    """Algorithmic tensor FLOPs of one call: (2K+1) * 2NVd."""
    return (2 * K + 1) * 2.0 * N * V * d


def kept_call_flops(n_kept, d: int, V: int) -> float:
    """Algorithmic tensor FLOPs spent on kept tokens only: 2r = 4Vd per kept
    token of an auxiliary module and 3r = 6Vd per kept token of the final one
    (``n_kept``: kept-token counts of the K modules, final module last).  The
    call itself still runs masked tokens through every product."""
    n = [int(x) for x in n_kept]
    return 4.0 * V * d * sum(n[:-1]) + 6.0 * V * d * n[-1]


def gemm_flops(M: int, N: int, Kdim: int) -> float:
    return 2.0 * M * N * Kdim


def min_bytes(K: int, N: int, d: int, V: int) -> int:
    """Compulsory HBM bytes of one call: H in, W in, dH out, dW out, targets, losses."""
    return K * N * d * 2 + V * d * 2 + K * N * d * 2 + V * d * 4 + K * N * 8
