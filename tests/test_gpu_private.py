"""GPU parity of private readouts (each module its own W_k and final-norm
gain gamma_k, with dW_k and dgamma_k) against the fp64 oracle."""
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


def _params(wl):
    """Distinct readouts and gains per module: the workload's generator with per-module seeds."""
    Ws = [synth.gen_W(wl.with_(seed=wl.seed + 100 * k)) for k in range(wl.K)]
    gs = [synth.gen_gamma(wl.with_(seed=wl.seed + 100 * k)) for k in range(wl.K)]
    return Ws, gs


@pytest.mark.parametrize("wl,with_heads", [
    (Workload("priv_k3_n200_d136_v1001", K=3, N=200, d=136, V=1001, seed=71, mask_frac=0.1,
              row_scale=True), False),
    (Workload("priv_k2_n256_d256_v2048_heads", K=2, N=256, d=256, V=2048, seed=72,
              heavy_frac=0.01), True),
], ids=["plain", "heads"])
def test_private_readouts(sr, wl, with_heads):
    import torch
    inp = synth.generate(wl)
    Ws, gs = _params(wl)
    K, N, d, V = wl.K, wl.N, wl.d, wl.V
    dev = torch.device("cuda")
    hidden = [parity.to_device_bf16(inp.hidden[k]) for k in range(K)]
    Wd = [parity.to_device_bf16(w) for w in Ws]
    gd = [parity.to_device_bf16(g) for g in gs]
    tg = torch.from_numpy(inp.targets).to(dev)
    loss_tok = torch.empty(K, N, device=dev)
    loss_mean = torch.empty(K, device=dev)
    dh = [torch.empty(N, d, dtype=torch.bfloat16, device=dev) for _ in range(K)]
    dW = [torch.empty(V, d, device=dev) for _ in range(K)]
    dg = [torch.empty(d, device=dev) for _ in range(K)]
    dims = sr.make_dims(K, N, d, V)
    ws = torch.empty(sr.solo_readout_private_workspace_bytes(dims), dtype=torch.uint8,
                     device=dev)
    heads = {}
    tau = bias = None
    if with_heads:
        tau, bias = synth.gen_heads(wl)
        heads = dict(tau=torch.from_numpy(tau).to(dev), bias=torch.from_numpy(bias).to(dev),
                     dtau=torch.empty(K, device=dev), dbias=torch.empty(K, V, device=dev))
    sr.solo_readout_fwd_bwd_private(dims, hidden, gd, Wd, tg, None, loss_tok, loss_mean, dh, dW,
                                    dg, ws, **heads)
    assert sr.solo_readout_get_flags(ws) == 0
    dec = orc.bf16_bits_to_f64
    ref = orc.solo_readout_private([dec(inp.hidden[k]) for k in range(K)],
                                   [dec(g) for g in gs], [dec(w) for w in Ws],
                                   inp.targets.astype(np.int64), eps=float(np.float32(wl.eps)),
                                   tau=None if tau is None else tau.astype(np.float64),
                                   bias=None if bias is None else bias.astype(np.float64))
    got = dict(loss_tok=loss_tok.double().cpu().numpy(),
               loss_mean=loss_mean.double().cpu().numpy(),
               dhidden=[parity.bf16_tensor_to_f64(x) for x in dh])
    rep = parity.compare_full(wl, got, ref, check_dW=False, check_dgamma=False)
    for k in range(K):
        parity.check_grad(f"dW[{k}]", dW[k].double().cpu().numpy(), ref["dW"][k], rep)
        parity.check_grad(f"dgamma[{k}]", dg[k].double().cpu().numpy(), ref["dgamma"][k], rep)
    if with_heads:
        parity.check_grad("dtau", heads["dtau"].double().cpu().numpy(), ref["dtau"], rep)
        for k in range(K):
            parity.check_grad(f"dbias[{k}]", heads["dbias"][k].double().cpu().numpy(),
                              ref["dbias"][k], rep)
    print(wl.name, rep)
