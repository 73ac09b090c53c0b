"""The final RMSNorm's quantisation is bit-exact against the oracle.

x-hat = bf16(gamma h r) is a quantised code, so both sides take the rounding
decision on the exact value: the oracle in fp64 (exact for these products to
far below the bf16 spacing), the GPU with an error-free fp32 sum of squares,
a refined reciprocal square root and an exact test of products near a bf16
midpoint.  Every bit of x-hat must agree, at the headline size too, where
thousands of products fall within 4 fp32 ulp of a midpoint and take the exact
test; r agrees to fp32 rounding.
"""
import numpy as np
import pytest

import oracle.solo_oracle as orc
from paper_2609_35440_gb300 import synth, workloads
from paper_2609_35440_gb300.workloads import Workload
from tests import parity

pytestmark = pytest.mark.gpu

SHAPES = [Workload("bits_k3_n200_d72_v1001", K=3, N=200, d=72, V=1001, seed=91, row_scale=True),
          Workload("bits_k2_n1_d8_v16", K=2, N=1, d=8, V=16, seed=92),
          Workload("bits_k2_n70_d2600_v600", K=2, N=70, d=2600, V=600, seed=93, row_scale=True),
          workloads.W1P3B]


@pytest.mark.parametrize("wl", SHAPES, ids=lambda w: w.name)
def test_xhat_bits_equal_the_oracle(wl):
    import torch
    from paper_2609_35440_gb300 import solo_readout as sr
    dims = sr.make_dims(wl.K, wl.N, wl.d, wl.V, wl.eps, wl.ignore_index)
    hid_bits = [synth.gen_hidden(wl, k) for k in range(wl.K)]
    gamma_bits = synth.gen_gamma(wl)
    hid = [parity.to_device_bf16(h) for h in hid_bits]
    xhat = torch.empty(wl.K * wl.N, wl.d, dtype=torch.bfloat16, device="cuda")
    r = torch.empty(wl.K * wl.N, dtype=torch.float32, device="cuda")
    sr.solo_readout_rmsnorm(dims, hid, parity.to_device_bf16(gamma_bits), xhat, r)
    torch.cuda.synchronize()
    got = xhat.view(torch.int16).cpu().numpy().view(np.uint16)
    got_r = r.cpu().numpy().astype(np.float64)
    dec = orc.bf16_bits_to_f64
    gamma = dec(gamma_bits)
    eps = float(np.float32(wl.eps))
    near = 0
    for k in range(wl.K):
        h = dec(hid_bits[k])
        rows = slice(k * wl.N, (k + 1) * wl.N)
        r_ref, xq = orc.rmsnorm_forward(h, gamma, eps, contract=True)
        want = synth.to_bf16_bits(xq)          # xq holds bf16 values: the conversion is exact
        bad = np.flatnonzero(got[rows] != want)
        assert bad.size == 0, (k, bad.size, bad[:5])
        assert np.max(np.abs(got_r[rows] - r_ref) / r_ref) <= 2e-7
        # products within 4 fp32 ulp of a bf16 midpoint: the exact-test path
        y32 = (gamma[None, :] * h * r_ref[:, None]).astype(np.float32).view(np.uint32)
        low = (y32 & np.uint32(0xFFFF)).astype(np.int64) - 0x8000
        near += int(np.sum(np.abs(low) <= 4))
    if wl.K * wl.N * wl.d >= 1 << 24:
        assert near > 1000, near
