"""Failure detection on the GPU without faulting it: the bounded wait used by
every pipeline role gives up on a barrier that nothing arrives on, the kernel
reports SOLO_FLAG_TIMEOUT and returns, and the context stays usable."""
import time

import numpy as np
import pytest

from paper_2609_35440_gb300 import synth, workloads
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


def test_wait_that_nothing_completes_times_out_and_returns(sr):
    import torch
    flags = torch.zeros(1, dtype=torch.int32, device="cuda")
    t = time.time()
    sr.solo_readout_selftest_wait_timeout(flags, 2000)        # 2 ms limit
    torch.cuda.synchronize()
    assert time.time() - t < 5.0
    assert int(flags.item()) == sr.SOLO_FLAG_TIMEOUT
    # the context is still usable: a normal call afterwards is correct and clean
    wl = workloads.SMOKE
    inp = synth.generate(wl)
    gpu = parity.run_gpu(wl, inp)
    assert gpu["flags"] == 0
    parity.compare_full(wl, gpu, parity.oracle_full(wl, inp))
