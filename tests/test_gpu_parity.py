"""GPU parity against the fp64 oracle, element by element, on sizes the
oracle finishes in seconds: the smallest workload, ragged shapes that leave
partial tiles in every dimension, masks, bad targets, optional outputs and
run-to-run determinism.  All calls go through the C ABI."""
import numpy as np
import pytest

from paper_2609_35440_gb300 import synth, workloads
from paper_2609_35440_gb300.workloads import Workload
from tests import parity

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda(built_library):
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_35440_gb300 import solo_readout
    solo_readout.load(built_library)


def _case(wl, mask=None, targets=None, **kw):
    inp = synth.generate(wl)
    gpu = parity.run_gpu(wl, inp, mask=mask, targets=targets, **kw)
    ref = parity.oracle_full(wl, inp, mask=mask, targets=targets)
    return inp, gpu, ref


def test_smallest_workload_full_parity():
    wl = workloads.SMOKE
    _, gpu, ref = _case(wl)
    rep = parity.compare_full(wl, gpu, ref)
    assert gpu["flags"] == 0
    print("report", rep)


RAGGED = [
    Workload("ragged_k3_n200_d72_v1001", K=3, N=200, d=72, V=1001, seed=31, mask_frac=0.1,
             row_scale=True),
    Workload("ragged_k2_n130_d264_v517", K=2, N=130, d=264, V=517, seed=32, heavy_frac=0.02),
    Workload("k1_n64_d128_v300", K=1, N=64, d=128, V=300, seed=33),
    Workload("k4_n33_d136_v4100_zipf", K=4, N=33, d=136, V=4100, seed=34, targets="zipf",
             mask_frac=0.2),
    Workload("k2_n1_d8_v16", K=2, N=1, d=8, V=16, seed=35),
    Workload("k2_n300_d512_v2500_heavy", K=2, N=300, d=512, V=2500, seed=36, heavy_frac=0.01,
             row_scale=True, mask_frac=0.05),
    # the largest module count the call takes (SOLO_MAX_MODULES)
    Workload("k16_n40_d64_v777", K=16, N=40, d=64, V=777, seed=37, mask_frac=0.05),
    # d above 2048: the row kernels' generic path (rows re-read instead of cached)
    Workload("k2_n70_d2600_v600", K=2, N=70, d=2600, V=600, seed=38, row_scale=True),
]


@pytest.mark.parametrize("wl", RAGGED, ids=lambda w: w.name)
def test_ragged_shapes(wl):
    _, gpu, ref = _case(wl)
    parity.compare_full(wl, gpu, ref)


# Vocabularies narrower than one 64-column TMA box and than the 16-byte row of
# the exponential buffer: the loads past V read zeros, the stores past V are
# dropped, and with V = 1 every loss and gradient is exactly zero.
TINY_V = [Workload(f"k2_n50_d64_v{V}", K=2, N=50, d=64, V=V, seed=60 + V, mask_frac=0.1)
          for V in (1, 3, 8, 13)]


@pytest.mark.parametrize("wl", TINY_V, ids=lambda w: w.name)
def test_tiny_vocabulary(wl):
    _, gpu, ref = _case(wl)
    assert gpu["flags"] == 0
    parity.compare_full(wl, gpu, ref)
    if wl.V == 1:
        assert not np.any(gpu["loss_tok"]) and not np.any(gpu["dW"])
        for k in range(wl.K):
            assert not np.any(gpu["dhidden"][k])


# Every GEMM runs several work units per CTA pair here (76 pairs on GB300), so
# the second TMEM accumulator, its phase flips and raster groups beyond the
# first are compared element by element:
#  - 4096 x 2 tokens, d = 1024, V = 8192: logits 32 x 32 = 1024 tiles, dX̂ 32 x 4 =
#    128 tiles (36 + 52 cut into 2 parts), dW 32 x 4 = 128 tiles;
#  - 3000 x 3 tokens, d = 776, V = 5000 (no dimension a multiple of 256): logits
#    36 x 20 = 720 tiles, dX̂ 36 x 4 = 144, dW 20 x 4 = 80 (4 tiles cut into 8).
MULTIWAVE = [
    Workload("k2_n4096_d1024_v8192_rowscale_zipf_mask10", K=2, N=4096, d=1024, V=8192,
             seed=51, targets="zipf", mask_frac=0.1, row_scale=True),
    Workload("k3_n3000_d776_v5000_heavy_mask5", K=3, N=3000, d=776, V=5000, seed=52,
             heavy_frac=0.01, mask_frac=0.05, row_scale=True),
]


# Masked tokens are skipped by every product (the kept ones are compacted into
# the first rows): most tokens masked, a final module with a few kept tokens
# whose compact rows start off a 32-row boundary, every token of a module kept.
MASKED = [
    Workload("k3_n700_d264_v1500_mask90", K=3, N=700, d=264, V=1500, seed=53, mask_frac=0.9,
             row_scale=True),
    Workload("k4_n2000_d512_v3000_mask37", K=4, N=2000, d=512, V=3000, seed=54,
             mask_frac=0.37, targets="zipf"),
]


@pytest.mark.parametrize("wl", MASKED, ids=lambda w: w.name)
def test_masked_tokens_skipped_full_parity(wl):
    _, gpu, ref = _case(wl)
    assert gpu["flags"] == 0
    parity.compare_full(wl, gpu, ref)


def test_all_tokens_masked():
    """Nothing kept anywhere: every loss and gradient is exactly zero."""
    wl = Workload("k2_n300_d128_v900_none", K=2, N=300, d=128, V=900, seed=55)
    inp = synth.generate(wl)
    tg = np.full_like(inp.targets, wl.ignore_index)
    gpu = parity.run_gpu(wl, inp, targets=tg)
    assert gpu["flags"] == 0
    assert not np.any(gpu["loss_tok"]) and not np.any(gpu["loss_mean"])
    for k in range(wl.K):
        assert not np.any(gpu["dhidden"][k])
    assert not np.any(gpu["dW"]) and not np.any(gpu["dgamma"])


@pytest.mark.parametrize("wl", MULTIWAVE, ids=lambda w: w.name)
def test_multiwave_full_parity(wl):
    """Element-by-element parity where every persistent GEMM loops over many
    tiles per CTA pair (both accumulators, raster groups, cut last waves)."""
    import torch
    from paper_2609_35440_gb300 import solo_readout as sr
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    pairs = sms // 2
    tiles = lambda rows, cols: -(-rows // 256) * -(-cols // 256)
    assert tiles(wl.M, wl.V) > 4 * pairs and tiles(wl.M, wl.d) > pairs
    assert tiles(wl.V, wl.d) > pairs
    _, gpu, ref = _case(wl)
    assert gpu["flags"] == 0
    rep = parity.compare_full(wl, gpu, ref)
    print(wl.name, rep)


def test_mask_array_and_bad_targets():
    wl = Workload("masked_k2_n160_d128_v700", K=2, N=160, d=128, V=700, seed=41)
    inp = synth.generate(wl)
    mask = synth.random_mask(7, wl.K, wl.N, 0.25)
    tg = inp.targets.copy()
    tg[0, 3] = wl.V           # out of range: masked and flagged
    tg[1, 9] = -7             # negative, not ignore_index: masked and flagged
    tg[1, 10] = wl.ignore_index
    gpu = parity.run_gpu(wl, inp, mask=mask, targets=tg)
    ref = parity.oracle_full(wl, inp, mask=mask, targets=tg)
    assert ref["bad_target"]
    assert gpu["flags"] & 1
    parity.compare_full(wl, gpu, ref)
    for k, n in ((0, 3), (1, 9), (1, 10)):
        assert gpu["loss_tok"][k, n] == 0.0
        assert not np.any(gpu["dhidden"][k][n])
    for k in range(wl.K):
        dead = mask[k] == 0
        assert np.all(gpu["loss_tok"][k][dead] == 0.0)
        assert not np.any(gpu["dhidden"][k][dead])


def test_module_without_kept_tokens():
    wl = Workload("allmasked_k2_n100_d64_v300", K=2, N=100, d=64, V=300, seed=42)
    inp = synth.generate(wl)
    tg = inp.targets.copy()
    tg[1, :] = wl.ignore_index       # final module: nothing kept
    gpu = parity.run_gpu(wl, inp, targets=tg)
    ref = parity.oracle_full(wl, inp, targets=tg)
    assert gpu["loss_mean"][1] == 0.0 and gpu["flags"] == 0
    assert not np.any(gpu["dhidden"][1]) and not np.any(gpu["dW"]) and not np.any(gpu["dgamma"])
    parity.compare_full(wl, gpu, ref)


def test_optional_outputs_and_determinism():
    wl = Workload("k3_n96_d192_v900", K=3, N=96, d=192, V=900, seed=43, mask_frac=0.1)
    inp = synth.generate(wl)
    a = parity.run_gpu(wl, inp)
    b = parity.run_gpu(wl, inp)
    for key in ("loss_tok", "loss_mean", "dW", "dgamma"):
        assert np.array_equal(a[key], b[key]), key
    for k in range(wl.K):
        assert np.array_equal(a["dhidden"][k], b["dhidden"][k])
    c = parity.run_gpu(wl, inp, want_dW=False, want_dgamma=False, want_loss_tok=False)
    assert np.array_equal(a["loss_mean"], c["loss_mean"])
    for k in range(wl.K):
        assert np.array_equal(a["dhidden"][k], c["dhidden"][k])


def test_workspace_reuse_across_shapes():
    """A workspace sized for a larger problem serves a smaller one; stale contents do not leak."""
    import torch
    from paper_2609_35440_gb300 import solo_readout as sr
    big = Workload("k2_n256_d256_v2048", K=2, N=256, d=256, V=2048, seed=44)
    small = Workload("k2_n100_d128_v1000", K=2, N=100, d=128, V=1000, seed=45, mask_frac=0.1)
    ws = torch.zeros(sr.solo_readout_workspace_bytes(sr.make_dims(big.K, big.N, big.d, big.V)),
                     dtype=torch.uint8, device="cuda")
    for wl in (big, small, big):
        inp = synth.generate(wl)
        gpu = parity.run_gpu(wl, inp)
        ro = gpu["_ro"]
        ro.workspace = ws
        hid = [parity.to_device_bf16(inp.hidden[k]) for k in range(wl.K)]
        ro(hid, parity.to_device_bf16(inp.gamma), parity.to_device_bf16(inp.W),
           torch.from_numpy(inp.targets).cuda())
        torch.cuda.synchronize()
        assert torch.equal(ro.loss_mean.cpu(), torch.from_numpy(gpu["loss_mean"]).float())


def test_kernel_launch_counter():
    """The library's launch counter sees every kernel of a call: the same call
    twice counts the same, the split last wave adds its fix-up kernels, and
    leaving out dW and dgamma removes their kernels."""
    import torch
    from paper_2609_35440_gb300 import solo_readout as sr
    wl = Workload("k2_n600_d256_v3000", K=2, N=600, d=256, V=3000, seed=46)
    inp = synth.generate(wl)
    hid = [parity.to_device_bf16(inp.hidden[k]) for k in range(wl.K)]
    gamma, W = parity.to_device_bf16(inp.gamma), parity.to_device_bf16(inp.W)
    tg = torch.from_numpy(inp.targets).cuda()

    def count(**kw):
        ro = sr.Readout(wl.K, wl.N, wl.d, wl.V, **kw)
        n0 = sr.solo_readout_kernel_launches()
        ro(hid, gamma, W, tg)
        n = sr.solo_readout_kernel_launches() - n0
        torch.cuda.synchronize()
        return n

    full = count()
    assert full == count()
    # kept-token scan and offsets, rmsnorm, logits, lse, module means, the
    # gradient pass's row classification and its whole rows, dxhat (with the
    # RMSNorm backward), dW, dgamma reduce: 11, plus the dW fix-up when its last
    # wave was cut and the RMSNorm backward of dX̂'s cut tiles
    assert 11 <= full <= 13
    # without dW and dgamma: no dW GEMM (nor its fix-up) and no dgamma reduction
    assert 9 <= count(want_dW=False, want_dgamma=False) <= full - 2


def test_zero_readout_closed_forms():
    """W = 0: every logit is 0, so each kept token's loss is ln V, dH and dgamma
    are exactly zero, and dW = (1/Nvalid) sum_i (1/V - e_{y_i}) xhat_i^T for the
    final module (the closed form, evaluated in fp64 from the GPU's own inputs)."""
    import oracle.solo_oracle as orc
    wl = Workload("zeroW_k2_n300_d136_v1001", K=2, N=300, d=136, V=1001, seed=47,
                  mask_frac=0.1)
    inp = synth.generate(wl)
    inp.W = np.zeros_like(inp.W)
    gpu = parity.run_gpu(wl, inp)
    assert gpu["flags"] == 0
    kept = inp.targets != wl.ignore_index
    lnV = np.log(wl.V)
    assert np.max(np.abs(gpu["loss_tok"][kept] - lnV)) <= 1e-5
    assert np.all(gpu["loss_tok"][~kept] == 0.0)
    assert np.allclose(gpu["loss_mean"], lnV, rtol=1e-6, atol=0.0)
    for k in range(wl.K):
        assert not np.any(gpu["dhidden"][k])
    assert not np.any(gpu["dgamma"])
    # dW of the final module from its x-hat (rounded exactly as the GPU rounds it)
    dec = orc.bf16_bits_to_f64
    k = wl.K - 1
    xhat = orc.rmsnorm_forward(dec(inp.hidden[k]), dec(inp.gamma), float(np.float32(wl.eps)),
                               contract=True)[1]
    y = inp.targets[k]
    keep = y != wl.ignore_index
    g = np.zeros((wl.N, wl.V))
    g[keep] = 1.0 / wl.V
    g[np.flatnonzero(keep), y[keep]] -= 1.0
    want = g.T @ xhat / keep.sum()
    parity.check_grad("dW (W = 0)", gpu["dW"], want, {})
