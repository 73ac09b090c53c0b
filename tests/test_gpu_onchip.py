"""GPU parity of solo_readout_fwd_bwd_onchip against the fp64 oracle.

The auxiliary modules run the single-pass on-chip kernel (the logits of a
128-row block and a 128-column vocabulary tile live in tensor and shared
memory only; a cluster of 1, 2, 4 or 8 CTAs splits d), the final module the
stored path.  The shapes below reach every cluster size, widths that leave
part or all of a CTA's slice past d, vocabularies that end inside a tile,
several row blocks per cluster, one module (nothing auxiliary) and sixteen,
masks and bad targets, a module with nothing kept, and rows whose logits
climb far above their first tile's maximum (the block is swept a second time
with the exact maximum).  All calls go through the C ABI."""
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


def _case(wl, mask=None, targets=None, inp=None):
    inp = synth.generate(wl) if inp is None else inp
    gpu = parity.run_gpu(wl, inp, mask=mask, targets=targets, onchip=True)
    ref = parity.oracle_full(wl, inp, mask=mask, targets=targets)
    return inp, gpu, ref


SHAPES = [
    workloads.SMOKE,                                                            # C = 1
    Workload("k3_n200_d72_v1001_ragged", K=3, N=200, d=72, V=1001, seed=61, mask_frac=0.1,
             row_scale=True),                                                   # C = 1, ds 128
    Workload("k3_n300_d512_v2500_heavy", K=3, N=300, d=512, V=2500, seed=62, heavy_frac=0.01,
             row_scale=True, mask_frac=0.05),                                   # C = 2
    Workload("k2_n1000_d1024_v3000_zipf", K=2, N=1000, d=1024, V=3000, seed=63,
             targets="zipf"),                                                   # C = 4
    Workload("k2_n600_d2048_v1500_rowscale", K=2, N=600, d=2048, V=1500, seed=64,
             row_scale=True, mask_frac=0.1),                                    # C = 8
    Workload("k2_n130_d776_v517", K=2, N=130, d=776, V=517, seed=65),           # C = 4, slice past d
    Workload("k2_n90_d520_v300", K=2, N=90, d=520, V=300, seed=66),             # C = 4, one CTA idle
    Workload("k1_n64_d128_v300", K=1, N=64, d=128, V=300, seed=67),             # no auxiliary module
    Workload("k16_n40_d64_v777", K=16, N=40, d=64, V=777, seed=68, mask_frac=0.05),
    Workload("k2_n1_d8_v16", K=2, N=1, d=8, V=16, seed=69),
    Workload("k3_n4096_d1024_v8192_multiblock", K=3, N=4096, d=1024, V=8192, seed=70,
             targets="zipf", mask_frac=0.1, row_scale=True),                    # 64 row blocks
]


TINY_V = [Workload(f"onchip_k2_n50_d64_v{V}", K=2, N=50, d=64, V=V, seed=80 + V, mask_frac=0.1)
          for V in (1, 3)]


@pytest.mark.parametrize("wl", TINY_V, ids=lambda w: w.name)
def test_onchip_tiny_vocabulary(wl):
    """One vocabulary tile, almost all of it past V: masked out of every sum."""
    _, gpu, ref = _case(wl)
    assert gpu["flags"] == 0
    parity.compare_full(wl, gpu, ref)


@pytest.mark.parametrize("wl", SHAPES, ids=lambda w: w.name)
def test_onchip_full_parity(wl):
    _, gpu, ref = _case(wl)
    assert gpu["flags"] == 0
    rep = parity.compare_full(wl, gpu, ref)
    print(wl.name, rep)


def test_onchip_matches_stored_path_and_is_deterministic():
    """Within the parity tolerances of the stored path's results (the
    exponentials use a different reference), and bitwise equal from call to call."""
    wl = Workload("k3_n500_d1024_v2000", K=3, N=500, d=1024, V=2000, seed=71, mask_frac=0.1)
    inp = synth.generate(wl)
    a = parity.run_gpu(wl, inp, onchip=True)
    b = parity.run_gpu(wl, inp, onchip=True)
    for key in ("loss_tok", "loss_mean", "dW", "dgamma"):
        assert np.array_equal(a[key], b[key]), key
    for k in range(wl.K):
        assert np.array_equal(a["dhidden"][k], b["dhidden"][k]), k
    st = parity.run_gpu(wl, inp)
    assert float(np.max(np.abs(a["loss_tok"] - st["loss_tok"]))) <= parity.LOSS_TOK_ABS
    rep = {}
    for k in range(wl.K):
        parity.check_grad(f"dH[{k}] vs stored", a["dhidden"][k], st["dhidden"][k], rep)
    # the final module takes the stored path on its own rows (its dgamma blocks of
    # 32 rows and its cut tiles fall differently): equal within the tolerances
    parity.check_grad("dW vs stored", a["dW"], st["dW"], rep)
    parity.check_grad("dgamma vs stored", a["dgamma"], st["dgamma"], rep)


def test_onchip_masks_bad_targets_and_empty_module():
    wl = Workload("masked_k3_n160_d256_v700", K=3, N=160, d=256, V=700, seed=72)
    inp = synth.generate(wl)
    mask = synth.random_mask(9, wl.K, wl.N, 0.25)
    tg = inp.targets.copy()
    tg[0, 3] = wl.V           # out of range: masked and flagged
    tg[0, 9] = -7             # negative, not ignore_index: masked and flagged
    tg[1, :] = wl.ignore_index          # module 1 (auxiliary): nothing kept
    _, gpu, ref = _case(wl, mask=mask, targets=tg)
    assert gpu["flags"] & 1
    assert gpu["loss_mean"][1] == 0.0 and not np.any(gpu["dhidden"][1])
    parity.compare_full(wl, gpu, ref)
    for k in range(wl.K):
        dead = (mask[k] == 0) | (tg[k] < 0) | (tg[k] >= wl.V)
        assert np.all(gpu["loss_tok"][k][dead] == 0.0)
        assert not np.any(gpu["dhidden"][k][dead])


def test_onchip_logits_far_above_the_first_tile():
    """Rows whose largest logit (in the last vocabulary tile) exceeds their first
    tile's maximum by about 90: the first sweep stops adding them and the block
    is swept again with the exact maximum as the reference."""
    wl = Workload("k2_n96_d64_v1000_climb", K=2, N=96, d=64, V=1000, seed=73)
    inp = synth.generate(wl)
    import oracle.solo_oracle as orc
    dec = orc.bf16_bits_to_f64
    W = dec(inp.W)
    gamma = dec(inp.gamma)
    # vocabulary entry 990 points along row 5 of module 0's normalised input, 990
    # and 991 along rows 7 and 50 of module 1 (a final-module row as well)
    for k, i, v in ((0, 5, 990), (0, 40, 991), (1, 7, 992)):
        h = dec(inp.hidden[k][i])
        xh = gamma * h / np.sqrt(np.mean(h * h) + wl.eps)
        W[v] = 11.5 * xh / np.linalg.norm(xh)
    inp.W = synth.to_bf16_bits(W)
    zmax = [float(np.max(orc.rmsnorm_forward(dec(inp.hidden[k]), gamma, wl.eps, True)[1][i]
                         @ dec(inp.W)[v])) for k, i, v in ((0, 5, 990), (0, 40, 991))]
    assert min(zmax) > 75.0, zmax
    tg = inp.targets.copy()
    tg[0, 40] = 991            # one climbing row predicts its own climbing entry
    _, gpu, ref = _case(wl, targets=tg, inp=inp)
    assert gpu["flags"] == 0
    assert np.all(np.isfinite(gpu["loss_tok"]))
    parity.compare_full(wl, gpu, ref)


FULL = [workloads.W340M, workloads.W1P3B, *workloads.SWEEP]


@pytest.mark.parametrize("wl", FULL, ids=lambda w: w.name)
def test_onchip_full_size_sampled_parity(wl):
    """The workloads of width <= 2048 at full size: sampled tokens of every
    module against the oracle one by one, the whole final module through the
    chunked oracle, and the module means against the token losses."""
    import torch
    inp = synth.generate(wl)
    gpu = parity.run_gpu(wl, inp, onchip=True)
    assert gpu["flags"] == 0
    rep = parity.sampled_check(wl, inp, gpu, full_final=True)
    print(wl.name, rep)
    del gpu
    torch.cuda.empty_cache()
