"""The checked build: every computed global index of the row kernels and the
GEMM epilogues is tested against its buffer (a violation sets
SOLO_FLAG_BOUNDS instead of making the access).  On ragged shapes that cut
the last wave of the backward products, with heads' parameters and through
the exit readout, it must set no flag and give bitwise the release build's
outputs.  Each library runs in its own process (the binding loads one)."""
import os
import subprocess
import sys

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SCRIPT = r"""
import sys
import numpy as np
import torch
sys.path.insert(0, sys.argv[2])
from paper_2609_35440_gb300 import solo_readout as sr, synth
from paper_2609_35440_gb300.workloads import Workload
from tests import parity

out = {"build_flags": np.array([sr.solo_readout_build_flags()])}
shapes = [Workload("ragged_k3_n200_d72_v1001", K=3, N=200, d=72, V=1001, seed=31,
                   mask_frac=0.1, row_scale=True),
          Workload("k2_n600_d256_v3000", K=2, N=600, d=256, V=3000, seed=46),
          Workload("k16_n40_d64_v777", K=16, N=40, d=64, V=777, seed=37, mask_frac=0.05),
          Workload("k2_n70_d2600_v600", K=2, N=70, d=2600, V=600, seed=38)]
for i, wl in enumerate(shapes):
    inp = synth.generate(wl)
    g = parity.run_gpu(wl, inp)
    out[f"{i}_flags"] = np.array([g["flags"]])
    for key in ("loss_tok", "loss_mean", "dW", "dgamma"):
        out[f"{i}_{key}"] = g[key]
    for k in range(wl.K):
        out[f"{i}_dh{k}"] = g["dhidden"][k]
    # heads' temperature and bias with their gradients
    tau, bias = synth.gen_heads(wl)
    hid = [parity.to_device_bf16(inp.hidden[k]) for k in range(wl.K)]
    gamma, W = parity.to_device_bf16(inp.gamma), parity.to_device_bf16(inp.W)
    tg = torch.from_numpy(inp.targets).cuda()
    ro = sr.Readout(wl.K, wl.N, wl.d, wl.V, eps=wl.eps)
    ro(hid, gamma, W, tg, tau=torch.from_numpy(tau).cuda(), bias=torch.from_numpy(bias).cuda(),
       head_grads=True)
    torch.cuda.synchronize()
    out[f"{i}_h_flags"] = np.array([ro.flags()])
    for key in ("loss_tok", "dW", "dgamma", "dtau", "dbias"):
        out[f"{i}_h_{key}"] = getattr(ro, key).cpu().numpy()
    # exit readout
    ex = sr.ExitReadout(wl.K, wl.N, wl.d, wl.V, eps=wl.eps)
    ex(hid, gamma, W, tg)
    torch.cuda.synchronize()
    out[f"{i}_x_flags"] = np.array([ex.flags()])
    out[f"{i}_x_top1"] = ex.top1.cpu().numpy()
    out[f"{i}_x_loss_tok"] = ex.loss_tok.cpu().numpy()
np.savez(sys.argv[1], **out)
"""


def _run(lib: str, dest: str) -> dict:
    env = dict(os.environ, SOLO_READOUT_LIB=lib)
    subprocess.run([sys.executable, "-c", SCRIPT, dest, ROOT], env=env, check=True, cwd=ROOT,
                   timeout=600)
    with np.load(dest) as f:
        return {k: f[k] for k in f.files}


def test_checked_build_matches_release(tmp_path, built_library):
    from paper_2609_35440_gb300 import build as b
    checked = b.LIB_CHECKED if b.up_to_date_checked() else b.build(checked=True)
    rel = _run(built_library, str(tmp_path / "release.npz"))
    chk = _run(checked, str(tmp_path / "checked.npz"))
    assert rel["build_flags"][0] == 0 and chk["build_flags"][0] == 1
    assert rel.keys() == chk.keys()
    for key in rel:
        if key.endswith("flags") and key != "build_flags":
            assert rel[key][0] == 0 and chk[key][0] == 0, (key, rel[key], chk[key])
        elif key != "build_flags":
            assert np.array_equal(rel[key], chk[key]), key
