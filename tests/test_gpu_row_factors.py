"""The auxiliary modules' gradient formed in the dX̂ epilogue.

The logits epilogue stores each tile's exponentials against the reference 0
while the tile's maximum logit stays within +-64.  A row all of whose tiles
did so (and whose log-sum-exp is at most 60) skips the gradient pass: the dX̂
epilogue forms tau/Nvalid (e^{-lse} (P W) - (1 - p_y) W_y) itself; a final-module
row gets its target entry of P and its x̂ row scaled instead (dW = P'^T (c x̂)).
The other rows go through the gradient pass.  These tests put auxiliary-module
rows in each regime and compare every output with the fp64 oracle:
  - logits about 90 above the rest (a tile stored against its own maximum);
  - every logit of a row below -64;
  - many logits near 60, so that lse exceeds 60 while every tile stays in bound;
  - confident rows, 1 - p_y of 1e-6 .. 1e-4, formed in the epilogue (each dH
    row compared on its own scale).
"""
import numpy as np
import pytest

import oracle.solo_oracle as orc
from paper_2609_35440_gb300 import synth
from paper_2609_35440_gb300.workloads import Workload
from tests import parity

pytestmark = pytest.mark.gpu

ROW_REL = 2e-2


@pytest.fixture(scope="module", autouse=True)
def _cuda(built_library):
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_35440_gb300 import solo_readout
    solo_readout.load(built_library)


def _xhat(wl, inp, k):
    dec = orc.bf16_bits_to_f64
    return orc.rmsnorm_forward(dec(inp.hidden[k]), dec(inp.gamma), float(np.float32(wl.eps)),
                               contract=True)[1]


def _check(wl, inp):
    gpu = parity.run_gpu(wl, inp)
    assert gpu["flags"] == 0
    ref = parity.oracle_full(wl, inp)
    parity.compare_full(wl, gpu, ref)
    return gpu, ref


def test_aux_rows_with_a_tile_far_above_zero():
    """Vocabulary rows 700 and 701 point along two rows of module 0 (an
    auxiliary module), with logits near 90 there."""
    wl = Workload("climb_k2_n96_d64_v1000", K=2, N=96, d=64, V=1000, seed=81)
    inp = synth.generate(wl)
    W = orc.bf16_bits_to_f64(inp.W)
    xh = _xhat(wl, inp, 0)
    for i, v in ((3, 700), (40, 701)):
        W[v] = 11.5 * xh[i] / np.linalg.norm(xh[i])
    inp.W = synth.to_bf16_bits(W)
    z = _xhat(wl, inp, 0) @ orc.bf16_bits_to_f64(inp.W).T
    assert z[3, 700] > 80 and z[40, 701] > 80
    inp.targets = inp.targets.copy()
    inp.targets[0, 40] = 701              # one of them predicts its climbing entry
    _check(wl, inp)


def test_aux_rows_with_every_logit_below_minus_64():
    """Module 0's rows share a direction u; every vocabulary row points against
    it, so all their logits lie near -80 (spread ~2.4 by the rows' own parts,
    which keeps the softmax from being flat: a flat one makes dH a difference
    of near-equal sums that the bf16 gradient cannot resolve)."""
    wl = Workload("sunk_k2_n64_d64_v600", K=2, N=64, d=64, V=600, seed=82)
    inp = synth.generate(wl)
    rng = np.random.default_rng(82)
    u = rng.standard_normal(wl.d)
    inp.hidden[0] = synth.to_bf16_bits(u[None, :] + 0.05 * rng.standard_normal((wl.N, wl.d)))
    xh = _xhat(wl, inp, 0)
    unit = u / np.linalg.norm(u)
    scale = 80.0 / float(np.mean(xh @ unit))
    W = -scale * unit[None, :] + 0.3 * rng.standard_normal((wl.V, wl.d))
    inp.W = synth.to_bf16_bits(W)
    z = _xhat(wl, inp, 0) @ orc.bf16_bits_to_f64(inp.W).T
    assert np.max(z) < -64, np.max(z)
    _check(wl, inp)


def test_aux_rows_with_log_sum_exp_above_60():
    """Half of the vocabulary gives module 0's rows logits near 55 (spread
    ~1.6, all below the bound of 64), so lse ~ 55 + ln(300) + 1.3 > 60."""
    wl = Workload("heavy_lse_k2_n64_d64_v600", K=2, N=64, d=64, V=600, seed=83)
    inp = synth.generate(wl)
    rng = np.random.default_rng(83)
    u = rng.standard_normal(wl.d)
    inp.hidden[0] = synth.to_bf16_bits(u[None, :] + 0.05 * rng.standard_normal((wl.N, wl.d)))
    xh = _xhat(wl, inp, 0)
    unit = u / np.linalg.norm(u)
    scale = 55.0 / float(np.mean(xh @ unit))
    W = 0.2 * rng.standard_normal((wl.V, wl.d))
    W[::2] += scale * unit[None, :]
    inp.W = synth.to_bf16_bits(W)
    z = _xhat(wl, inp, 0) @ orc.bf16_bits_to_f64(inp.W).T
    lse = np.log(np.sum(np.exp(z - z.max(axis=1, keepdims=True)), axis=1)) + z.max(axis=1)
    assert np.max(z) < 64 and np.min(lse) > 60, (np.max(z), np.min(lse))
    _check(wl, inp)


def test_confident_aux_rows_formed_in_the_epilogue():
    """Module 0 (auxiliary) predicts target 0 with 1 - p_y of 1e-6 .. 1e-4."""
    wl = Workload("confident_aux_k2_n64_d128_v512", K=2, N=64, d=128, V=512, seed=84)
    inp = synth.generate(wl)
    rng = np.random.default_rng(84)
    u = rng.standard_normal(wl.d)
    inp.hidden[0] = synth.to_bf16_bits(u[None, :] + 0.3 * rng.standard_normal((wl.N, wl.d)))
    W = orc.bf16_bits_to_f64(inp.W)
    xh = _xhat(wl, inp, 0)
    unit = u / np.linalg.norm(u)
    W[0] = 17.0 / float(np.mean(xh @ unit)) * unit
    inp.W = synth.to_bf16_bits(W)
    inp.targets = inp.targets.copy()
    inp.targets[0, :] = 0
    gpu, ref = _check(wl, inp)
    one_minus_py = -np.expm1(-ref["loss_tok"][0])
    assert np.all(one_minus_py < 1e-4) and np.all(one_minus_py > 1e-7), one_minus_py
    worst = 0.0
    for i in range(wl.N):
        sc = np.max(np.abs(ref["dhidden"][0][i]))
        worst = max(worst, float(np.max(np.abs(gpu["dhidden"][0][i] - ref["dhidden"][0][i])) / sc))
    assert worst <= ROW_REL, worst
