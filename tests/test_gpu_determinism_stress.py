"""Repeated calls at full size give bit-identical outputs.

Every reduction of the library runs in a fixed order, so any difference
between two calls on the same inputs would be a race: an accumulator in
tensor memory reused before its epilogue finished reading it, a stage of the
operand ring refilled before its MMAs completed, or rows of the gradient
pass's list processed twice or not at all.  The call runs back to back many
times (at full size, so that every persistent GEMM runs many work units per
CTA pair, in the plain and the heads' mode and the on-chip call, whose
clusters exchange partial logits through distributed shared memory) and each
output is compared on the device with the first call's.
"""
import numpy as np
import pytest

from paper_2609_35440_gb300 import synth, workloads
from tests import parity

pytestmark = pytest.mark.gpu

CALLS = 40


@pytest.fixture(scope="module")
def sr(built_library):
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_35440_gb300 import solo_readout
    solo_readout.load(built_library)
    return solo_readout


def _outputs(ro, heads):
    outs = [ro.loss_tok, ro.loss_mean, ro.dW, ro.dgamma, *ro.dhidden]
    if heads:
        outs += [ro.dtau, ro.dbias]
    return [t.clone() for t in outs]


@pytest.mark.parametrize("mode", ["plain", "heads", "onchip"])
def test_back_to_back_calls_are_bitwise_equal(sr, mode):
    import torch
    wl = workloads.W1P3B
    inp = synth.generate(wl)
    hidden = [parity.to_device_bf16(inp.hidden[k]) for k in range(wl.K)]
    gamma, W = parity.to_device_bf16(inp.gamma), parity.to_device_bf16(inp.W)
    tg = torch.from_numpy(np.ascontiguousarray(inp.targets, dtype=np.int32)).cuda()
    heads = mode == "heads"
    kw = {}
    if heads:
        tau, bias = synth.gen_heads(wl)
        kw = dict(tau=torch.from_numpy(tau).cuda(), bias=torch.from_numpy(bias).cuda(),
                  head_grads=True)
    ro = sr.Readout(wl.K, wl.N, wl.d, wl.V, eps=wl.eps, onchip=mode == "onchip")
    ro(hidden, gamma, W, tg, **kw)
    first = _outputs(ro, heads)
    mismatches = torch.zeros(len(first), dtype=torch.int64, device="cuda")
    for _ in range(CALLS):
        ro(hidden, gamma, W, tg, **kw)
        for i, (a, b) in enumerate(zip(first, _outputs(ro, heads))):
            mismatches[i] += (a.view(torch.uint8) != b.view(torch.uint8)).any().to(torch.int64)
    torch.cuda.synchronize()
    assert ro.flags() == 0
    assert not bool(mismatches.any()), mismatches.tolist()
