"""The allocation-free entry point, solo_readout_fwd_bwd_static.

Some callers cannot allocate device memory (a host that lets them enqueue
work but never allocate, or a loop whose memory was fixed at start-up), so
they cannot hand the library a workspace.  For them the library carries a
fixed 64 MiB scratch array of its own.  These tests call that entry point
through the C ABI and check, on two calls in a row with different shapes
(so the second call meets the first call's leftovers in the shared
scratch), that its outputs are bitwise those of the workspace entry point
(the same kernels run on the same inputs, so any difference would be stale
scratch leaking into a result), that both match the fp64 oracle element by
element within the parity tolerances, and that an oversized problem is
refused before any work is enqueued.  This file is collected last on purpose.
"""
import numpy as np
import pytest

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


def _static_call(sr, wl, inp):
    import torch
    dev = torch.device("cuda")
    hidden = [parity.to_device_bf16(inp.hidden[k]) for k in range(wl.K)]
    gamma = parity.to_device_bf16(inp.gamma)
    W = parity.to_device_bf16(inp.W)
    targets = torch.from_numpy(np.ascontiguousarray(inp.targets, np.int32)).to(dev)
    loss_tok = torch.full((wl.K, wl.N), float("nan"), device=dev)
    loss_mean = torch.full((wl.K,), float("nan"), device=dev)
    dhidden = [torch.empty(wl.N, wl.d, dtype=torch.bfloat16, device=dev) for _ in range(wl.K)]
    dW = torch.empty(wl.V, wl.d, dtype=torch.float32, device=dev)
    dgamma = torch.empty(wl.d, dtype=torch.float32, device=dev)
    flags = torch.full((1,), 0xFFFF, dtype=torch.int32, device=dev)
    dims = sr.make_dims(wl.K, wl.N, wl.d, wl.V, wl.eps, wl.ignore_index)
    sr.solo_readout_fwd_bwd_static(dims, hidden, gamma, W, targets, None, loss_tok, loss_mean,
                                   dhidden, dW, dgamma, device_flags=flags)
    torch.cuda.synchronize()
    return dict(loss_tok=loss_tok.double().cpu().numpy(),
                loss_mean=loss_mean.double().cpu().numpy(),
                dhidden=[parity.bf16_tensor_to_f64(x) for x in dhidden],
                dW=dW.double().cpu().numpy(), dgamma=dgamma.double().cpu().numpy(),
                flags=int(flags.item()))


def test_static_scratch_matches_workspace_entry_point(sr):
    shapes = [workloads.SMOKE,
              Workload("ragged_k3_n200_d72_v1001", K=3, N=200, d=72, V=1001, seed=31,
                       mask_frac=0.1, row_scale=True)]
    for wl in shapes:                       # two calls in a row on the shared scratch
        inp = synth.generate(wl)
        ref = parity.run_gpu(wl, inp)       # the workspace entry point
        got = _static_call(sr, wl, inp)
        assert got["flags"] == 0
        for key in ("loss_tok", "loss_mean", "dW", "dgamma"):
            assert np.array_equal(got[key], ref[key]), key
        for k in range(wl.K):
            assert np.array_equal(got["dhidden"][k], ref["dhidden"][k]), k
        # and both against the oracle, element by element
        parity.compare_full(wl, got, parity.oracle_full(wl, inp))


def test_static_scratch_rejects_oversized_problem(sr):
    import ctypes
    dims = sr.make_dims(4, 8192, 2048, 32000)
    assert sr.solo_readout_workspace_bytes(dims) > sr.SOLO_STATIC_SCRATCH_BYTES
    fake = 1 << 20                          # never dereferenced: refused on the host
    st = sr.solo_readout_fwd_bwd_static(dims, [fake] * 4, fake, fake, fake, None, None, fake,
                                        [fake] * 4, None, None, check=False)
    assert st == sr.SOLO_ERR_EXCEEDS_STATIC_SCRATCH
    assert "64 MiB" in sr.strerror(st)
