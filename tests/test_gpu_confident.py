"""Confident rows: every token of the final module has its target's
probability within ~1e-5 of 1.  Two quantities then cancel if formed
naively: p_y - 1 in the logit gradient, and E_p[s] - s_y, which gives the
RMSNorm backward's row sum in the dX̂ epilogue.  Each dH row is compared with
the fp64 oracle on its own scale, not only against the largest row of the
tensor, and dgamma and the losses are compared as in the other parity tests.
"""
import numpy as np
import pytest

import oracle.solo_oracle as orc
from paper_2609_35440_gb300 import synth
from paper_2609_35440_gb300.workloads import Workload
from tests import parity

pytestmark = pytest.mark.gpu

ROW_REL = 2e-2      # per row: max |gpu - oracle| / max |oracle| over the row


def confident_inputs(margin: float, shift: float = 0.0):
    """Module 1's hidden rows share a direction u; W's row 0 points along u
    with a length chosen so that its logit exceeds the others by ~margin;
    every target of module 1 is 0.  Module 0 is left as generated.  A shift
    moves every vocabulary row against u, lowering module 1's logits by
    ~shift."""
    wl = Workload("confident_k2_n64_d128_v512", K=2, N=64, d=128, V=512, seed=91)
    inp = synth.generate(wl)
    rng = np.random.default_rng(91)
    u = rng.standard_normal(wl.d)
    h = u[None, :] + 0.3 * rng.standard_normal((wl.N, wl.d))
    inp.hidden[1] = synth.to_bf16_bits(h)
    W = orc.bf16_bits_to_f64(inp.W)
    gamma = orc.bf16_bits_to_f64(inp.gamma)
    hb = orc.bf16_bits_to_f64(inp.hidden[1])
    r = 1.0 / np.sqrt(np.mean(hb * hb, axis=1) + wl.eps)
    xhat = gamma[None, :] * hb * r[:, None]
    unit = u / np.linalg.norm(u)
    beta = margin / float(np.mean(xhat @ unit))
    W[0] = beta * unit
    if shift:
        W = W - (shift / float(np.mean(xhat @ unit))) * unit[None, :]
    inp.W = synth.to_bf16_bits(W)
    inp.targets = inp.targets.copy()
    inp.targets[1, :] = 0
    return wl, inp


def test_confident_rows_keep_relative_precision():
    wl, inp = confident_inputs(margin=17.0)
    gpu = parity.run_gpu(wl, inp)
    assert gpu["flags"] == 0
    ref = parity.oracle_full(wl, inp)
    # the regime the test is about: 1 - p_y of 1e-6 .. 1e-4 on module 1
    lse = ref["loss_tok"][1]                      # loss = lse - z_y = -log p_y
    one_minus_py = -np.expm1(-lse)
    assert np.all(one_minus_py < 1e-4) and np.all(one_minus_py > 1e-7), one_minus_py
    dh_g, dh_r = gpu["dhidden"][1], ref["dhidden"][1]
    worst = 0.0
    for i in range(wl.N):
        scale = np.max(np.abs(dh_r[i]))
        assert scale > 0
        worst = max(worst, float(np.max(np.abs(dh_g[i] - dh_r[i])) / scale))
    assert worst <= ROW_REL, worst
    parity.compare_full(wl, gpu, ref)


def test_confident_rows_below_the_reference():
    """The same confident rows with every logit of module 1 about 25 lower: the
    target's logit (about -8) is the row's maximum but lies below the
    reference 0 that the exponentials of tiles within +-64 are stored against,
    so lse - z_y must come from log1p of the other terms relative to z_y."""
    wl, inp = confident_inputs(margin=17.0, shift=25.0)
    dec = orc.bf16_bits_to_f64
    xh = orc.rmsnorm_forward(dec(inp.hidden[1]), dec(inp.gamma), float(np.float32(wl.eps)),
                             contract=True)[1]
    z = xh @ dec(inp.W).T
    assert np.all(np.argmax(z, axis=1) == 0) and np.all(z[:, 0] < -2), z[:, 0]
    assert np.all(np.max(np.abs(z), axis=1) < 64)
    gpu = parity.run_gpu(wl, inp)
    assert gpu["flags"] == 0
    ref = parity.oracle_full(wl, inp)
    one_minus_py = -np.expm1(-ref["loss_tok"][1])
    assert np.all(one_minus_py < 1e-4) and np.all(one_minus_py > 1e-8), one_minus_py
    # the token losses themselves on their own scale (-log p_y ~ 1 - p_y): the
    # form (0 - z_y) + log(s + e^{z_y}) would be off by ~2e-2 here
    rel = np.abs(gpu["loss_tok"][1] - ref["loss_tok"][1]) / ref["loss_tok"][1]
    assert np.max(rel) <= 1e-3, float(np.max(rel))
    dh_g, dh_r = gpu["dhidden"][1], ref["dhidden"][1]
    worst = 0.0
    for i in range(wl.N):
        scale = np.max(np.abs(dh_r[i]))
        assert scale > 0
        worst = max(worst, float(np.max(np.abs(dh_g[i] - dh_r[i])) / scale))
    assert worst <= ROW_REL, worst
    parity.compare_full(wl, gpu, ref)
