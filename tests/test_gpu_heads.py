"""GPU parity of the call with each head's temperature tau_k and bias b_k
(Algorithm 1's local objective) against the fp64 oracle: losses, dH, dW,
dgamma, dtau and dbias, on small ragged shapes element by element and on a
340M-scale workload with every module's tau and bias gradients checked in
full through a chunked oracle."""
import numpy as np
import pytest

import oracle.solo_oracle as orc
from paper_2609_35440_gb300 import synth, workloads
from paper_2609_35440_gb300.workloads import Workload
from tests import parity

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sr(built_library):
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_35440_gb300 import solo_readout
    solo_readout.load(built_library)
    return solo_readout


def _gpu(sr, wl, inp, tau, bias, grads=True):
    import torch
    hidden = [parity.to_device_bf16(inp.hidden[k]) for k in range(wl.K)]
    gamma, W = parity.to_device_bf16(inp.gamma), parity.to_device_bf16(inp.W)
    tg = torch.from_numpy(inp.targets).cuda()
    ro = sr.Readout(wl.K, wl.N, wl.d, wl.V, eps=wl.eps)
    t = None if tau is None else torch.from_numpy(tau).cuda()
    b = None if bias is None else torch.from_numpy(bias).cuda()
    ro(hidden, gamma, W, tg, tau=t, bias=b, head_grads=grads)
    torch.cuda.synchronize()
    out = dict(loss_tok=ro.loss_tok.double().cpu().numpy(),
               loss_mean=ro.loss_mean.double().cpu().numpy(),
               dhidden=[parity.bf16_tensor_to_f64(x) for x in ro.dhidden],
               dW=ro.dW.double().cpu().numpy(), dgamma=ro.dgamma.double().cpu().numpy(),
               flags=ro.flags())
    if grads:
        out["dtau"] = ro.dtau.double().cpu().numpy()
        out["dbias"] = ro.dbias.double().cpu().numpy()
    return out


SMALL = [Workload("heads_k2_n256_d128_v4096", K=2, N=256, d=128, V=4096, seed=61),
         Workload("heads_k3_n200_d72_v1001", K=3, N=200, d=72, V=1001, seed=62, mask_frac=0.1,
                  row_scale=True),
         Workload("heads_k2_n300_d512_v2500_heavy", K=2, N=300, d=512, V=2500, seed=63,
                  heavy_frac=0.01, mask_frac=0.05)]


@pytest.mark.parametrize("wl", SMALL, ids=lambda w: w.name)
def test_heads_small_full_parity(sr, wl):
    inp = synth.generate(wl)
    tau, bias = synth.gen_heads(wl)
    gpu = _gpu(sr, wl, inp, tau, bias)
    assert gpu["flags"] == 0
    dec = orc.bf16_bits_to_f64
    ref = orc.solo_readout_fwd_bwd([dec(inp.hidden[k]) for k in range(wl.K)], dec(inp.gamma),
                                   dec(inp.W), inp.targets.astype(np.int64),
                                   eps=float(np.float32(wl.eps)), tau=tau.astype(np.float64),
                                   bias=bias.astype(np.float64))
    rep = parity.compare_full(wl, gpu, ref)
    parity.check_grad("dtau", gpu["dtau"], ref["dtau"], rep)
    for k in range(wl.K):
        parity.check_grad(f"dbias[{k}]", gpu["dbias"][k], ref["dbias"][k], rep)
    print(wl.name, rep)


@pytest.mark.parametrize("neg_tau,bias_std", [(True, 0.5), (False, 25.0)],
                         ids=["negative_tau", "wide_bias"])
def test_heads_reference_choices(sr, neg_tau, bias_std):
    """Temperatures of both signs (the first pass bounds tau s from the other
    side), and biases spanning far more than 60 within a tile (the first pass
    falls back to forming every z), both against the oracle."""
    wl = Workload("heads_k3_n200_d136_v1001", K=3, N=200, d=136, V=1001, seed=64,
                  mask_frac=0.05)
    inp = synth.generate(wl)
    tau, bias = synth.gen_heads(wl, bias_std=bias_std)
    if neg_tau:
        tau[0] = -0.7
    else:   # the tiles' bias spans exceed 60
        assert np.min(np.ptp(bias[:, :256], axis=1)) > 60.0
    gpu = _gpu(sr, wl, inp, tau, bias)
    assert gpu["flags"] == 0
    dec = orc.bf16_bits_to_f64
    ref = orc.solo_readout_fwd_bwd([dec(inp.hidden[k]) for k in range(wl.K)], dec(inp.gamma),
                                   dec(inp.W), inp.targets.astype(np.int64),
                                   eps=float(np.float32(wl.eps)), tau=tau.astype(np.float64),
                                   bias=bias.astype(np.float64))
    rep = parity.compare_full(wl, gpu, ref)
    parity.check_grad("dtau", gpu["dtau"], ref["dtau"], rep)
    for k in range(wl.K):
        parity.check_grad(f"dbias[{k}]", gpu["dbias"][k], ref["dbias"][k], rep)


def test_without_heads_is_the_plain_call_bitwise(sr):
    """tau = 1 and b = 0 give the plain call's results bit for bit.  With the
    bias gradient requested the bias-gradient pass sums every row's G and
    rewrites the rows without per-row factors in its own order of rounding
    (tau applied last), so the gradients then agree within the parity
    tolerances and the losses still bit for bit."""
    wl = SMALL[1]
    inp = synth.generate(wl)
    plain = parity.run_gpu(wl, inp)
    ones = np.ones(wl.K, np.float32)
    zeros = np.zeros((wl.K, wl.V), np.float32)
    for tau, bias, grads in ((None, None, False), (ones, zeros, False), (ones, zeros, True)):
        got = _gpu(sr, wl, inp, tau, bias, grads=grads)
        for key in ("loss_tok", "loss_mean"):
            assert np.array_equal(got[key], plain[key]), (key, grads)
        if grads:
            rep = {}
            parity.check_grad("dW", got["dW"], plain["dW"], rep)
            parity.check_grad("dgamma", got["dgamma"], plain["dgamma"], rep)
            for k in range(wl.K):
                parity.check_grad(f"dH[{k}]", got["dhidden"][k], plain["dhidden"][k], rep)
        else:
            for key in ("dW", "dgamma"):
                assert np.array_equal(got[key], plain[key]), key
            for k in range(wl.K):
                assert np.array_equal(got["dhidden"][k], plain["dhidden"][k]), k


def test_heads_340m_scale_every_module(sr):
    wl = workloads.W340M
    inp = synth.generate(wl)
    tau, bias = synth.gen_heads(wl)
    gpu = _gpu(sr, wl, inp, tau, bias)
    assert gpu["flags"] == 0
    dec = orc.bf16_bits_to_f64
    gamma, W = dec(inp.gamma), dec(inp.W)
    eps = float(np.float32(wl.eps))
    rep = {}
    dtau = np.zeros(wl.K)
    rng = np.random.default_rng(5)
    for k in range(wl.K):
        y = inp.targets[k].astype(np.int64)
        kept, _ = orc.kept_tokens(y, None, wl.V, wl.ignore_index)
        nv = int(kept.sum())
        db = np.zeros(wl.V)
        loss = np.zeros(wl.N)
        rows = rng.choice(wl.N, 24, replace=False)
        for i0 in range(0, wl.N, 512):
            sl = slice(i0, min(wl.N, i0 + 512))
            res = orc.module_rows(dec(inp.hidden[k][sl]), gamma, W, y[sl], kept[sl], nv, eps,
                                  True, tau=float(tau[k]), b=bias[k].astype(np.float64))
            dtau[k] += res["dtau"]
            db += res["db"]
            loss[sl] = res["loss"]
            sel = [r - i0 for r in rows if i0 <= r < sl.stop]
            if sel:
                parity.check_grad(f"dH[{k}] rows {i0}", gpu["dhidden"][k][i0 + np.array(sel)],
                                  res["dh"][sel], rep)
        assert np.max(np.abs(gpu["loss_tok"][k] - loss)) <= parity.LOSS_TOK_ABS
        want = loss.sum() / nv
        assert abs(gpu["loss_mean"][k] - want) <= parity.LOSS_MEAN_REL * abs(want)
        parity.check_grad(f"dbias[{k}]", gpu["dbias"][k], db, rep)
    parity.check_grad("dtau", gpu["dtau"], dtau, rep)
    print({key: v for key, v in rep.items() if "rows" not in key})
