"""Every workspace byte a call reads is written earlier in the same call, and
every output element is written (not accumulated).

The workspace and the outputs are filled with 0xFF bytes (NaN in bf16 and
fp32, -1 in int32) before the call.  With masked tokens in every module, the
kept tokens' compact rows start the final module at an offset that is not a
multiple of the 128-row reduction blocks, so the dW product's last block
reaches past the final module's kept rows: those rows must be zeros written by
the gradient pass, not what an earlier call left there.  Checked for the plain
call (rows whose gradient is P times a per-row factor), for the heads' call
with the bias gradient, for a second call on the same workspace with a
different mask, and for the on-chip call and the exit readout.
"""
import numpy as np
import pytest

import oracle.solo_oracle as orc
from paper_2609_35440_gb300 import synth
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


def _poison(ro):
    import torch
    ro.workspace.fill_(0xFF)
    for t in [ro.loss_tok, ro.loss_mean, ro.dW, ro.dgamma, ro.dtau, ro.dbias, *ro.dhidden]:
        t.view(torch.uint8).fill_(0xFF)


def _call(sr, wl, inp, ro, tau=None, bias=None):
    import torch
    hidden = [parity.to_device_bf16(inp.hidden[k]) for k in range(wl.K)]
    gamma, W = parity.to_device_bf16(inp.gamma), parity.to_device_bf16(inp.W)
    tg = torch.from_numpy(np.ascontiguousarray(inp.targets, dtype=np.int32)).cuda()
    t = None if tau is None else torch.from_numpy(tau).cuda()
    b = None if bias is None else torch.from_numpy(bias).cuda()
    heads = tau is not None
    ro(hidden, gamma, W, tg, tau=t, bias=b, head_grads=heads)
    torch.cuda.synchronize()
    out = dict(loss_tok=ro.loss_tok.double().cpu().numpy(),
               loss_mean=ro.loss_mean.double().cpu().numpy(),
               dhidden=[parity.bf16_tensor_to_f64(x) for x in ro.dhidden],
               dW=ro.dW.double().cpu().numpy(), dgamma=ro.dgamma.double().cpu().numpy(),
               flags=ro.flags())
    if heads:
        out["dtau"] = ro.dtau.double().cpu().numpy()
        out["dbias"] = ro.dbias.double().cpu().numpy()
    return out


def _oracle(wl, inp, tau=None, bias=None):
    dec = orc.bf16_bits_to_f64
    return orc.solo_readout_fwd_bwd(
        [dec(inp.hidden[k]) for k in range(wl.K)], dec(inp.gamma), dec(inp.W),
        inp.targets.astype(np.int64), eps=float(np.float32(wl.eps)),
        tau=None if tau is None else tau.astype(np.float64),
        bias=None if bias is None else bias.astype(np.float64), contract=True)


def _offsets(wl, inp):
    kept = (inp.targets != wl.ignore_index).sum(axis=1)
    return np.concatenate([[0], np.cumsum(kept)])


WL = Workload("stale_k3_n300_d192_v1800_mask30", K=3, N=300, d=192, V=1800, seed=91,
              mask_frac=0.3)


def test_plain_call_on_a_poisoned_workspace(sr):
    inp = synth.generate(WL)
    off = _offsets(WL, inp)
    assert off[WL.K - 1] % 128 != 0 and off[WL.K] - off[WL.K - 1] < WL.N
    ro = sr.Readout(WL.K, WL.N, WL.d, WL.V, eps=WL.eps)
    _poison(ro)
    gpu = _call(sr, WL, inp, ro)
    assert gpu["flags"] == 0
    parity.compare_full(WL, gpu, _oracle(WL, inp))


def test_heads_call_with_bias_gradient_on_a_poisoned_workspace(sr):
    inp = synth.generate(WL)
    tau, bias = synth.gen_heads(WL)
    ro = sr.Readout(WL.K, WL.N, WL.d, WL.V, eps=WL.eps)
    _poison(ro)
    gpu = _call(sr, WL, inp, ro, tau, bias)
    assert gpu["flags"] == 0
    ref = _oracle(WL, inp, tau, bias)
    rep = parity.compare_full(WL, gpu, ref)
    parity.check_grad("dtau", gpu["dtau"], ref["dtau"], rep)
    for k in range(WL.K):
        parity.check_grad(f"dbias[{k}]", gpu["dbias"][k], ref["dbias"][k], rep)


def test_second_call_with_fewer_kept_tokens(sr):
    """The first call keeps every token (its rows fill the whole buffer); the
    second masks 30% of them, so its tail rows hold the first call's data."""
    inp = synth.generate(WL)
    full = synth.generate(WL)
    full.targets = np.where(full.targets == WL.ignore_index, 1, full.targets).astype(
        full.targets.dtype)
    ro = sr.Readout(WL.K, WL.N, WL.d, WL.V, eps=WL.eps)
    _poison(ro)
    first = _call(sr, WL, full, ro)
    assert first["flags"] == 0
    gpu = _call(sr, WL, inp, ro)
    assert gpu["flags"] == 0
    parity.compare_full(WL, gpu, _oracle(WL, inp))


def test_onchip_call_on_a_poisoned_workspace(sr):
    inp = synth.generate(WL)
    ro = sr.Readout(WL.K, WL.N, WL.d, WL.V, eps=WL.eps, onchip=True)
    _poison(ro)
    gpu = _call(sr, WL, inp, ro)
    assert gpu["flags"] == 0
    parity.compare_full(WL, gpu, _oracle(WL, inp))


def test_exit_readout_on_a_poisoned_workspace(sr):
    import torch
    from tests.test_gpu_exit import _compare
    inp = synth.generate(WL)
    ex = sr.ExitReadout(WL.K, WL.N, WL.d, WL.V, eps=WL.eps)
    ex.workspace.fill_(0xFF)
    for t in (ex.loss_tok, ex.loss_mean, ex.top1, ex.top1_logprob):
        t.view(torch.uint8).fill_(0xFF)
    hidden = [parity.to_device_bf16(inp.hidden[k]) for k in range(WL.K)]
    gamma, W = parity.to_device_bf16(inp.gamma), parity.to_device_bf16(inp.W)
    tg = torch.from_numpy(np.ascontiguousarray(inp.targets, dtype=np.int32)).cuda()
    ex(hidden, gamma, W, tg)
    torch.cuda.synchronize()
    gpu = dict(top1=ex.top1.cpu().numpy(), top1_logprob=ex.top1_logprob.double().cpu().numpy(),
               loss_tok=ex.loss_tok.double().cpu().numpy(),
               loss_mean=ex.loss_mean.double().cpu().numpy(), flags=ex.flags())
    assert gpu["flags"] == 0
    _compare(WL, inp, gpu)
    np.testing.assert_allclose(gpu["loss_mean"], _oracle(WL, inp)["loss_mean"], rtol=1e-5, atol=0)
