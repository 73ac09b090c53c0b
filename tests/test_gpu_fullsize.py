"""GPU parity at the full workload sizes, in the launch configuration the
benchmark times: sampled tokens and vocabulary rows against the fp64 oracle,
the whole final module (mean loss, dgamma) through the chunked oracle, and
properties that hold at any size (module mean = mean of token losses, dW
columns sum to zero)."""
import pytest

from paper_2609_35440_gb300 import synth, workloads
from tests import parity

pytestmark = pytest.mark.gpu

FULL = [workloads.W340M, workloads.W1P3B, *workloads.SWEEP, workloads.W2B]


@pytest.fixture(scope="module", autouse=True)
def _cuda(built_library):
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_35440_gb300 import solo_readout
    solo_readout.load(built_library)


@pytest.mark.parametrize("wl", FULL, ids=lambda w: w.name)
def test_full_size_sampled_parity(wl):
    import torch
    inp = synth.generate(wl)
    gpu = parity.run_gpu(wl, inp)
    assert gpu["flags"] == 0
    rep = parity.sampled_check(wl, inp, gpu, full_final=True)
    print(wl.name, rep)
    del gpu
    torch.cuda.empty_cache()
