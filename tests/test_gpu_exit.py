"""GPU parity of the early-exit readout (forward only) against the oracle.

Losses and top-1 log-probabilities within the token-loss tolerance.  The
top-1 index is an argmax taken on fp32 logits on the GPU and fp64 logits in
the oracle, so it is compared where it is unique (the oracle's margin between
its best and second-best logit exceeds the fp32 accuracy of a logit) and
checked to be a valid maximum elsewhere."""
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


def _gpu_exit(sr, wl, inp, with_targets=True, mask=None):
    import torch
    hidden = [parity.to_device_bf16(inp.hidden[k]) for k in range(wl.K)]
    gamma, W = parity.to_device_bf16(inp.gamma), parity.to_device_bf16(inp.W)
    tg = torch.from_numpy(inp.targets).cuda() if with_targets else None
    mk = None if mask is None else torch.from_numpy(mask).cuda()
    ex = sr.ExitReadout(wl.K, wl.N, wl.d, wl.V, eps=wl.eps, with_targets=with_targets)
    ex(hidden, gamma, W, tg, mk)
    torch.cuda.synchronize()
    out = dict(top1=ex.top1.cpu().numpy(), top1_logprob=ex.top1_logprob.double().cpu().numpy(),
               flags=ex.flags())
    if with_targets:
        out["loss_tok"] = ex.loss_tok.double().cpu().numpy()
        out["loss_mean"] = ex.loss_mean.double().cpu().numpy()
    return out


def _check_top1(top1_gpu, z, report, key):
    """Unique where the oracle's margin exceeds the fp32 logit accuracy; valid elsewhere."""
    zmax = np.max(z, axis=1)
    tol = 1e-3 * np.maximum(1.0, np.abs(zmax))
    rows = np.arange(z.shape[0])
    part = np.partition(z, -2, axis=1)
    margin = part[:, -1] - part[:, -2]
    unique = margin > tol
    want = np.argmax(z, axis=1)
    assert np.array_equal(top1_gpu[unique], want[unique]), key
    assert np.all(z[rows, top1_gpu] >= zmax - tol), key
    report[key] = float(np.mean(unique))


def _compare(wl, inp, gpu, mask=None, rows=None):
    dec = orc.bf16_bits_to_f64
    rep = {}
    for k in range(wl.K):
        sel = np.arange(wl.N) if rows is None else rows
        h = dec(inp.hidden[k][sel])
        ref = orc.exit_readout([h], dec(inp.gamma), dec(inp.W),
                               None if "loss_tok" not in gpu else inp.targets[k:k + 1, sel],
                               None if mask is None else mask[k:k + 1, sel],
                               eps=float(np.float32(wl.eps)), contract=True)
        _check_top1(gpu["top1"][k][sel], ref["z"][0], rep, f"top1[{k}]")
        err = np.max(np.abs(gpu["top1_logprob"][k][sel] - ref["top1_logprob"][0]))
        assert err <= parity.LOSS_TOK_ABS, ("top1_logprob", k, err)
        if "loss_tok" in gpu:
            err = np.max(np.abs(gpu["loss_tok"][k][sel] - ref["loss_tok"][0]))
            assert err <= parity.LOSS_TOK_ABS, ("loss_tok", k, err)
            rep[f"loss_tok[{k}]"] = float(err)
    return rep


SMALL = [workloads.SMOKE,
         Workload("ragged_k3_n200_d72_v1001", K=3, N=200, d=72, V=1001, seed=31, mask_frac=0.1,
                  row_scale=True),
         Workload("k2_n300_d512_v2500_heavy", K=2, N=300, d=512, V=2500, seed=36,
                  heavy_frac=0.01, row_scale=True, mask_frac=0.05)]


TINY_V = [Workload(f"exit_k2_n50_d64_v{V}", K=2, N=50, d=64, V=V, seed=70 + V, mask_frac=0.1)
          for V in (2, 3, 13)]


@pytest.mark.parametrize("wl", TINY_V, ids=lambda w: w.name)
def test_exit_readout_tiny_vocabulary(sr, wl):
    """Vocabularies narrower than one 32-column chunk of the epilogue."""
    inp = synth.generate(wl)
    gpu = _gpu_exit(sr, wl, inp)
    assert gpu["flags"] == 0
    _compare(wl, inp, gpu)
    assert np.all((gpu["top1"] >= 0) & (gpu["top1"] < wl.V))


@pytest.mark.parametrize("wl", SMALL, ids=lambda w: w.name)
def test_exit_readout_small(sr, wl):
    inp = synth.generate(wl)
    gpu = _gpu_exit(sr, wl, inp)
    assert gpu["flags"] == 0
    _compare(wl, inp, gpu)
    # module means equal those of the training call, which tests pin in full
    train = parity.run_gpu(wl, inp)
    np.testing.assert_allclose(gpu["loss_mean"], train["loss_mean"], rtol=1e-6, atol=0)


def test_exit_readout_without_targets_and_with_mask(sr):
    wl = Workload("k2_n160_d128_v700", K=2, N=160, d=128, V=700, seed=51)
    inp = synth.generate(wl)
    plain = _gpu_exit(sr, wl, inp, with_targets=False)
    _compare(wl, inp, plain)
    mask = synth.random_mask(9, wl.K, wl.N, 0.3)
    gpu = _gpu_exit(sr, wl, inp, mask=mask)
    _compare(wl, inp, gpu, mask=mask)
    assert np.array_equal(gpu["top1"], plain["top1"])   # decoding ignores targets and masks
    assert np.all(gpu["loss_tok"][mask == 0] == 0.0)


@pytest.mark.parametrize("wl", [workloads.W1P3B, workloads.SWEEP[2]], ids=lambda w: w.name)
def test_exit_readout_full_size_sampled(sr, wl):
    inp = synth.generate(wl)
    gpu = _gpu_exit(sr, wl, inp)
    assert gpu["flags"] == 0
    rows = np.unique(np.concatenate([[0, wl.N - 1],
                                     np.random.default_rng(3).choice(wl.N, 48, replace=False)]))
    rep = _compare(wl, inp, gpu, rows=rows)
    for k in range(wl.K):   # module mean = mean of the kept token losses
        kept, _ = orc.kept_tokens(inp.targets[k], None, wl.V, wl.ignore_index)
        want = gpu["loss_tok"][k][kept].sum() / kept.sum()
        assert abs(gpu["loss_mean"][k] - want) <= 1e-6 * want
    print(wl.name, rep)


def test_exit_top1_ties_take_the_first_index(sr):
    """Readout rows copied to later positions (within a 32-column chunk, across
    chunks of a tile and across 256-column tiles) give exactly equal logits on
    the GPU; the top-1 is then the lowest index among the tied copies (the first
    maximum).  The oracle's logits are made exactly tied the same way (a copy
    takes its source's value) before its first argmax is taken."""
    wl = Workload("ties_k2_n256_d128_v1001", K=2, N=256, d=128, V=1001, seed=52)
    inp = synth.generate(wl)
    W = inp.W.copy()
    root = np.arange(wl.V)
    for dst, src in ((np.arange(1, 256, 2), np.arange(0, 256, 2)),     # same chunk
                     (np.arange(256, 512), np.arange(0, 256)),         # next tile
                     (np.arange(700, 740), np.arange(600, 640))):      # other chunks, tiles
        W[dst] = W[src]
        root[dst] = root[src]
    inp.W = W
    gpu = _gpu_exit(sr, wl, inp, with_targets=False)
    assert gpu["flags"] == 0
    dec = orc.bf16_bits_to_f64
    ties_seen = 0
    for k in range(wl.K):
        ref = orc.exit_readout([dec(inp.hidden[k])], dec(inp.gamma), dec(W), None, None,
                               eps=float(np.float32(wl.eps)), contract=True)
        z = ref["z"][0][:, root]                  # copies take exactly their source's value
        want = np.argmax(z, axis=1)               # first maximum
        best_root = root[want]
        other = np.where(root[None, :] == best_root[:, None], -np.inf, z)
        zmax = z[np.arange(wl.N), want]
        clear = zmax - other.max(axis=1) > 1e-3 * np.maximum(1.0, np.abs(zmax))
        assert np.array_equal(gpu["top1"][k][clear], want[clear])
        ties_seen += int(np.sum(clear & (np.sum(z == zmax[:, None], axis=1) > 1)))
    assert ties_seen > 0
