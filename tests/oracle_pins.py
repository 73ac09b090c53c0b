"""Pins of the fp64 oracle against facts that do not come from the oracle.

Each ``pin_*`` function raises AssertionError when the oracle disagrees with
a closed form, an invariant, brute force, finite differences or an
independent PyTorch fp64 composition.  ``test_oracle_pins.py`` runs them on
the oracle as written, and ``test_oracle_mutations.py`` runs them on copies
of the oracle with a planted mistake to show that each mistake is caught.
"""
from __future__ import annotations

import math

import numpy as np

from paper_2609_35440_gb300 import synth
from paper_2609_35440_gb300.workloads import Workload


def problem(K=2, N=6, d=8, V=16, seed=11, mask_frac=0.0, row_scale=False,
            heavy=0.0, targets="uniform", keep_mask=None, orc=None):
    """A small fp64 problem decoded from the seeded bf16 generator."""
    wl = Workload("pin", K=K, N=N, d=d, V=V, seed=seed, mask_frac=mask_frac,
                  row_scale=row_scale, heavy_frac=heavy, targets=targets)
    inp = synth.generate(wl)
    dec = orc.bf16_bits_to_f64
    hidden = [dec(inp.hidden[k]) for k in range(K)]
    return dict(hidden=hidden, gamma=dec(inp.gamma), W=dec(inp.W),
                targets=inp.targets.astype(np.int64), mask=keep_mask,
                eps=wl.eps, V=V, d=d, K=K, N=N)


def run(orc, p, contract=False, **kw):
    args = dict(hidden=p["hidden"], gamma=p["gamma"], W=p["W"],
                targets=p["targets"], mask=p["mask"], eps=p["eps"],
                contract=contract)
    args.update(kw)
    return orc.solo_readout_fwd_bwd(**args)


def rel(a, b):
    a, b = np.asarray(a, float), np.asarray(b, float)
    den = np.max(np.abs(b))
    return float(np.max(np.abs(a - b)) / (den if den > 0 else 1.0))


# -- bf16 rounding ------------------------------------------------------------

def pin_bf16_rounding(orc):
    q = orc.round_to_bf16
    cases = [
        (1.0, 1.0),
        (1.0 + 2.0 ** -8, 1.0),                       # tie -> even (down)
        (1.0 + 3 * 2.0 ** -8, 1.0 + 2.0 ** -6),      # tie -> even (up)
        (1.0 + 2.0 ** -8 + 2.0 ** -40, 1.0 + 2.0 ** -7),  # above tie: up
        (-(1.0 + 2.0 ** -8), -1.0),
        (3.0 * 2.0 ** 20 + 2.0 ** 13, 3.0 * 2.0 ** 20),  # 8 significant bits
        (255.5, 256.0),                               # tie at 9 bits -> even
        (254.5, 254.0),
        (0.0, 0.0),
        (1.0 / 3.0, 0.333984375),
    ]
    for x, want in cases:
        got = float(q(np.array([x]))[0])
        assert got == want, (x, got, want)


# -- loss ---------------------------------------------------------------------

def pin_zero_readout(orc):
    """W = 0: loss = ln V exactly, dH = dgamma = 0, dW in closed form."""
    p = problem(K=2, N=7, d=8, V=24, seed=3, mask_frac=0.3, orc=orc)
    p["W"] = np.zeros_like(p["W"])
    for contract in (False, True):
        out = run(orc, p, contract=contract)
        K, V = p["K"], p["V"]
        kept, _ = orc.kept_tokens(p["targets"][K - 1], None, V, -100)
        for k in range(K):
            kk, _ = orc.kept_tokens(p["targets"][k], None, V, -100)
            np.testing.assert_allclose(out["loss_tok"][k][kk], math.log(V), rtol=0, atol=1e-13)
            assert np.all(out["loss_tok"][k][~kk] == 0.0)
            np.testing.assert_allclose(out["loss_mean"][k], math.log(V), rtol=0, atol=1e-13)
            assert np.all(out["dhidden"][k] == 0.0)
        assert np.all(out["dgamma"] == 0.0)
        # closed form: dW = (1/Nvalid) sum_i (1/V - e_{y_i}) xhat_i^T
        h = p["hidden"][K - 1]
        ms = np.array([sum(v * v for v in row) / p["d"] for row in h])
        xhat = p["gamma"][None, :] * h / np.sqrt(ms + p["eps"])[:, None]
        if contract:
            xhat = orc.round_to_bf16(xhat)
        nv = kept.sum()
        want = np.zeros((V, p["d"]))
        for i in np.nonzero(kept)[0]:
            want += xhat[i][None, :] / V
            want[p["targets"][K - 1][i]] -= xhat[i]
        want /= nv
        np.testing.assert_allclose(out["dW"], want, rtol=1e-12, atol=1e-15)


def pin_brute_force_ce(orc):
    """Per-token CE from explicit loops, no max shift, small logits."""
    p = problem(K=1, N=5, d=6, V=12, seed=5, orc=orc)
    p["W"] = p["W"] * 10.0          # logits of order one
    out = run(orc, p, contract=False)
    h, g, W = p["hidden"][0], p["gamma"], p["W"]
    d, V = p["d"], p["V"]
    for i in range(p["N"]):
        ms = sum(h[i][j] ** 2 for j in range(d)) / d
        r = 1.0 / math.sqrt(ms + p["eps"])
        x = [g[j] * h[i][j] * r for j in range(d)]
        z = [sum(x[j] * W[v][j] for j in range(d)) for v in range(V)]
        want = math.log(sum(math.exp(zv) for zv in z)) - z[p["targets"][0][i]]
        assert abs(out["loss_tok"][0][i] - want) < 1e-12, (i, out["loss_tok"][0][i], want)


# -- gradients ----------------------------------------------------------------

def _loss_k(orc, p, k, **over):
    q = dict(p)
    q.update(over)
    return run(orc, q, contract=False)["loss_mean"][k]


def pin_finite_differences(orc):
    """Central differences of the module losses (exact mode, fp64)."""
    p = problem(K=2, N=4, d=8, V=16, seed=7, mask_frac=0.25, row_scale=True, orc=orc)
    p["W"] = p["W"] * 20.0
    out = run(orc, p, contract=False)
    K, step = p["K"], 1e-6
    for k in range(K):
        num = np.zeros_like(p["hidden"][k])
        for idx in np.ndindex(*num.shape):
            hp = [h.copy() for h in p["hidden"]]
            hm = [h.copy() for h in p["hidden"]]
            hp[k][idx] += step
            hm[k][idx] -= step
            num[idx] = (_loss_k(orc, p, k, hidden=hp) - _loss_k(orc, p, k, hidden=hm)) / (2 * step)
        assert rel(out["dhidden"][k], num) < 1e-7, ("dH", k, rel(out["dhidden"][k], num))
    numW = np.zeros_like(p["W"])
    for idx in np.ndindex(*numW.shape):
        Wp, Wm = p["W"].copy(), p["W"].copy()
        Wp[idx] += step
        Wm[idx] -= step
        numW[idx] = (_loss_k(orc, p, K - 1, W=Wp) - _loss_k(orc, p, K - 1, W=Wm)) / (2 * step)
    assert rel(out["dW"], numW) < 1e-7, ("dW", rel(out["dW"], numW))
    numg = np.zeros_like(p["gamma"])
    for j in range(len(numg)):
        gp, gm = p["gamma"].copy(), p["gamma"].copy()
        gp[j] += step
        gm[j] -= step
        numg[j] = (_loss_k(orc, p, K - 1, gamma=gp) - _loss_k(orc, p, K - 1, gamma=gm)) / (2 * step)
    assert rel(out["dgamma"], numg) < 1e-7, ("dgamma", rel(out["dgamma"], numg))


def pin_softmax_rows_sum_to_zero(orc):
    """Rows of (softmax - onehot) sum to zero; adding a common row to W changes nothing."""
    p = problem(K=2, N=9, d=16, V=40, seed=9, mask_frac=0.2, orc=orc)
    p["W"] = p["W"] * 30.0
    out = run(orc, p, contract=False)
    for res in out["rows"]:
        assert np.max(np.abs(res["g"].sum(axis=1))) < 1e-15
    c = np.linspace(-0.5, 0.7, p["d"])
    out2 = run(orc, dict(p, W=p["W"] + c[None, :]), contract=False)
    for k in range(p["K"]):
        np.testing.assert_allclose(out2["loss_tok"][k], out["loss_tok"][k], rtol=0, atol=1e-11)
        assert rel(out2["dhidden"][k], out["dhidden"][k]) < 1e-9
    # each column of dW sums to zero over the vocabulary
    colsum = out["dW"].sum(axis=0)
    assert np.max(np.abs(colsum)) < 1e-14 * max(1.0, np.max(np.abs(out["dW"])))


def pin_scale_invariance(orc):
    """With eps = 0 the loss is degree-0 homogeneous in h: dH(a h) = dH(h)/a and <dh_i, h_i> = 0."""
    p = problem(K=1, N=6, d=16, V=32, seed=13, orc=orc)
    p["W"] = p["W"] * 10.0
    p["eps"] = 0.0
    out = run(orc, p, contract=False)
    a = 3.7
    out2 = run(orc, dict(p, hidden=[h * a for h in p["hidden"]]), contract=False)
    np.testing.assert_allclose(out2["loss_tok"], out["loss_tok"], rtol=1e-12, atol=1e-13)
    assert rel(out2["dhidden"][0] * a, out["dhidden"][0]) < 1e-11
    dh, h = out["dhidden"][0], p["hidden"][0]
    euler = np.abs(np.sum(dh * h, axis=1)) / (np.linalg.norm(dh, axis=1) * np.linalg.norm(h, axis=1))
    assert np.max(euler) < 1e-12


def pin_masking(orc):
    """Masked tokens: zero loss and an exactly-zero dH row; out of range = masked + flagged."""
    p = problem(K=2, N=8, d=8, V=16, seed=15, orc=orc)
    keep = np.ones((2, 8), dtype=np.uint8)
    keep[0, [1, 5]] = 0
    p["mask"] = keep
    tg = p["targets"].copy()
    tg[1, 2] = -100
    tg[1, 6] = 16            # out of range -> masked and flagged
    p["targets"] = tg
    out = run(orc, p, contract=True)
    assert out["bad_target"]
    for k, rows in ((0, [1, 5]), (1, [2, 6])):
        assert np.all(out["loss_tok"][k][rows] == 0.0)
        assert np.all(out["dhidden"][k][rows] == 0.0)
        assert out["n_valid"][k] == 6
        kept = np.ones(8, bool)
        kept[rows] = False
        np.testing.assert_allclose(out["loss_mean"][k], out["loss_tok"][k][kept].mean(), rtol=1e-14)
    # a module with no kept token: zero loss, zero gradients
    p["targets"] = np.full_like(tg, -100)
    out = run(orc, p, contract=True)
    assert np.all(out["loss_mean"] == 0.0) and not out["bad_target"]
    assert all(np.all(dh == 0.0) for dh in out["dhidden"])
    assert np.all(out["dW"] == 0.0) and np.all(out["dgamma"] == 0.0)


def pin_dgamma_identity(orc):
    """sum_j gamma_j dgamma_j = sum_i <dxhat_i, xhat_i> (exact mode)."""
    p = problem(K=2, N=10, d=16, V=32, seed=17, row_scale=True, orc=orc)
    p["W"] = p["W"] * 10.0
    out = run(orc, p, contract=False)
    res = out["rows"][-1]
    lhs = float(np.dot(p["gamma"], out["dgamma"]))
    rhs = float(np.sum(res["dxhat"] * res["xhat"]))
    assert abs(lhs - rhs) <= 1e-12 * max(1.0, abs(rhs)), (lhs, rhs)


def pin_torch_fp64(orc):
    """Independent composition of library routines: F.rms_norm, matmul, F.cross_entropy, autograd."""
    import torch
    import torch.nn.functional as F
    p = problem(K=3, N=11, d=24, V=50, seed=19, mask_frac=0.2, row_scale=True,
                heavy=0.1, orc=orc)
    p["W"] = p["W"] * 5.0
    out = run(orc, p, contract=False)
    W = torch.tensor(p["W"], dtype=torch.float64, requires_grad=True)
    g = torch.tensor(p["gamma"], dtype=torch.float64, requires_grad=True)
    for k in range(p["K"]):
        h = torch.tensor(p["hidden"][k], dtype=torch.float64, requires_grad=True)
        y = torch.tensor(p["targets"][k], dtype=torch.int64)
        x = F.rms_norm(h, (p["d"],), weight=g, eps=p["eps"])
        loss = F.cross_entropy(x @ W.T, y, ignore_index=-100)
        W.grad = None
        g.grad = None
        loss.backward()
        assert abs(loss.item() - out["loss_mean"][k]) < 1e-12
        assert rel(out["dhidden"][k], h.grad.numpy()) < 1e-11
        if k == p["K"] - 1:
            assert rel(out["dW"], W.grad.numpy()) < 1e-11
            assert rel(out["dgamma"], g.grad.numpy()) < 1e-11


def pin_row_subsets(orc):
    """module_rows on a subset and the chunked final-module pass agree with the full oracle."""
    p = problem(K=2, N=37, d=16, V=64, seed=21, mask_frac=0.2, orc=orc)
    out = run(orc, p, contract=True)
    k = 1
    kept, _ = orc.kept_tokens(p["targets"][k], None, p["V"], -100)
    rows = np.array([0, 5, 17, 36])
    sub = orc.module_rows(p["hidden"][k][rows], p["gamma"], p["W"], p["targets"][k][rows],
                          kept[rows], int(kept.sum()), p["eps"], True)
    np.testing.assert_allclose(sub["loss"], out["loss_tok"][k][rows], rtol=1e-15, atol=0)
    np.testing.assert_allclose(sub["dh"], out["dhidden"][k][rows], rtol=1e-15, atol=0)
    cols = np.array([0, 3, 63])
    ch = orc.final_module_chunked(lambda i0, n: p["hidden"][k][i0:i0 + n], p["N"], p["gamma"],
                                  p["W"], p["targets"][k], kept, p["eps"], True, dW_cols=cols,
                                  chunk=8)
    np.testing.assert_allclose(ch["loss"], out["loss_tok"][k], rtol=1e-14, atol=1e-15)
    np.testing.assert_allclose(ch["dgamma"], out["dgamma"], rtol=1e-12, atol=1e-18)
    np.testing.assert_allclose(ch["dW_rows"], out["dW"][cols], rtol=1e-12, atol=1e-18)


def pin_init_statistics(orc):
    """At init, lse_i = ln V + sigma_i^2/2 to first order with sigma_i^2 = |xhat_i|^2 E[W^2],
    and the mean loss differs from the mean lse by the mean target logit, which is
    zero-mean with spread sigma/sqrt(N)."""
    p = problem(K=1, N=256, d=256, V=2048, seed=23, orc=orc)
    out = run(orc, p, contract=True)
    res = out["rows"][0]
    s2 = np.sum(res["xhat"] ** 2, axis=1) * np.mean(p["W"] ** 2)
    want = math.log(p["V"]) + s2 / 2.0
    assert np.max(np.abs(res["lse"] - want)) < 0.2 * np.max(s2) ** 2 + 0.02, np.max(np.abs(res["lse"] - want))
    assert abs(np.mean(res["lse"]) - np.mean(want)) < 0.01
    spread = math.sqrt(float(np.mean(s2)) / p["N"])
    assert abs(out["loss_mean"][0] - np.mean(res["lse"])) < 4 * spread


PINS = [pin_bf16_rounding, pin_zero_readout, pin_brute_force_ce, pin_finite_differences,
        pin_softmax_rows_sum_to_zero, pin_scale_invariance, pin_masking, pin_dgamma_identity,
        pin_torch_fp64, pin_row_subsets, pin_init_statistics]


# -- early-exit readout ---------------------------------------------------------

def pin_exit_readout(orc):
    """Exits: brute-force argmax and log-probabilities; W = 0 decodes index 0 with
    log p = -ln V; p(top1) >= p(y) with equality when the target is the argmax;
    its losses equal the training call's."""
    p = problem(K=2, N=6, d=8, V=20, seed=25, mask_frac=0.2, orc=orc)
    p["W"] = p["W"] * 40.0
    ex = orc.exit_readout(p["hidden"], p["gamma"], p["W"], p["targets"], eps=p["eps"],
                          contract=False)
    for k in range(p["K"]):
        h = p["hidden"][k]
        for i in range(p["N"]):
            ms = sum(v * v for v in h[i]) / p["d"]
            r = 1.0 / math.sqrt(ms + p["eps"])
            x = [p["gamma"][j] * h[i][j] * r for j in range(p["d"])]
            z = [sum(x[j] * p["W"][v][j] for j in range(p["d"])) for v in range(p["V"])]
            best = max(range(p["V"]), key=lambda v: (z[v], -v))
            assert ex["top1"][k][i] == best
            lse = math.log(sum(math.exp(zv) for zv in z))
            assert abs(ex["top1_logprob"][k][i] - (z[best] - lse)) < 1e-12
            y = p["targets"][k][i]
            if y >= 0:
                assert ex["top1_logprob"][k][i] >= -ex["loss_tok"][k][i] - 1e-12
                if y == best:
                    assert abs(ex["top1_logprob"][k][i] + ex["loss_tok"][k][i]) < 1e-12
    full = run(orc, p, contract=False)
    np.testing.assert_allclose(ex["loss_tok"], full["loss_tok"], rtol=0, atol=1e-13)
    np.testing.assert_allclose(ex["loss_mean"], full["loss_mean"], rtol=0, atol=1e-13)
    z0 = orc.exit_readout(p["hidden"], p["gamma"], np.zeros_like(p["W"]), None,
                          eps=p["eps"], contract=True)
    assert np.all(z0["top1"] == 0)
    np.testing.assert_allclose(z0["top1_logprob"], -math.log(p["V"]), rtol=0, atol=1e-13)


PINS.append(pin_exit_readout)


# -- heads' temperature and bias ------------------------------------------------

def _heads(p, seed=0):
    rng = np.random.default_rng(seed)
    tau = 0.5 + rng.random(p["K"])
    bias = rng.normal(0.0, 0.7, size=(p["K"], p["V"]))
    return tau, bias


def pin_heads_finite_differences(orc):
    """Central differences of every module loss in tau_k, b_k, h_k, and of the final
    loss in W and gamma, with non-trivial temperatures and biases (exact mode)."""
    p = problem(K=2, N=4, d=8, V=12, seed=27, mask_frac=0.25, row_scale=True, orc=orc)
    p["W"] = p["W"] * 20.0
    tau, bias = _heads(p, 1)
    base = dict(tau=tau, bias=bias)
    out = run(orc, p, contract=False, **base)
    K, step = p["K"], 1e-6

    def L(k, **over):
        kw = dict(base)
        kw.update({x: v for x, v in over.items() if x in ("tau", "bias")})
        q = dict(p)
        q.update({x: v for x, v in over.items() if x not in ("tau", "bias")})
        return run(orc, q, contract=False, **kw)["loss_mean"][k]

    for k in range(K):
        tp, tm = tau.copy(), tau.copy()
        tp[k] += step
        tm[k] -= step
        num = (L(k, tau=tp) - L(k, tau=tm)) / (2 * step)
        assert abs(out["dtau"][k] - num) <= 1e-7 * max(1.0, abs(num)), ("dtau", k, out["dtau"][k], num)
        numb = np.zeros(p["V"])
        for v in range(p["V"]):
            bp, bm = bias.copy(), bias.copy()
            bp[k, v] += step
            bm[k, v] -= step
            numb[v] = (L(k, bias=bp) - L(k, bias=bm)) / (2 * step)
        assert rel(out["dbias"][k], numb) < 1e-7, ("dbias", k, rel(out["dbias"][k], numb))
        numh = np.zeros_like(p["hidden"][k])
        for idx in np.ndindex(*numh.shape):
            hp = [h.copy() for h in p["hidden"]]
            hm = [h.copy() for h in p["hidden"]]
            hp[k][idx] += step
            hm[k][idx] -= step
            numh[idx] = (L(k, hidden=hp) - L(k, hidden=hm)) / (2 * step)
        assert rel(out["dhidden"][k], numh) < 1e-7, ("dH", k)
    numW = np.zeros_like(p["W"])
    for idx in np.ndindex(*numW.shape):
        Wp, Wm = p["W"].copy(), p["W"].copy()
        Wp[idx] += step
        Wm[idx] -= step
        numW[idx] = (L(K - 1, W=Wp) - L(K - 1, W=Wm)) / (2 * step)
    assert rel(out["dW"], numW) < 1e-7, ("dW", rel(out["dW"], numW))


def pin_heads_closed_forms(orc):
    """W = 0: z = b, so loss = lse(b) - b_y, dtau = 0, db = mean over kept tokens of
    softmax(b) - e_y; each db_k sums to zero; a constant added to b_k changes nothing."""
    p = problem(K=2, N=9, d=8, V=16, seed=29, mask_frac=0.2, orc=orc)
    tau, bias = _heads(p, 2)
    p0 = dict(p, W=np.zeros_like(p["W"]))
    out = run(orc, p0, contract=True, tau=tau, bias=bias)
    for k in range(p["K"]):
        kept, _ = orc.kept_tokens(p["targets"][k], None, p["V"], -100)
        b = bias[k]
        lse_b = math.log(sum(math.exp(x) for x in b))
        prob = np.array([math.exp(x - lse_b) for x in b])
        y = p["targets"][k]
        for i in range(p["N"]):
            want = lse_b - b[y[i]] if kept[i] else 0.0
            assert abs(out["loss_tok"][k][i] - want) < 1e-12
        assert abs(out["dtau"][k]) < 1e-15
        want_db = np.zeros(p["V"])
        for i in np.nonzero(kept)[0]:
            want_db += prob
            want_db[y[i]] -= 1.0
        want_db /= kept.sum()
        np.testing.assert_allclose(out["dbias"][k], want_db, rtol=0, atol=1e-13)
    out = run(orc, p, contract=False, tau=tau, bias=bias)
    assert np.max(np.abs(out["dbias"].sum(axis=1))) < 1e-14
    shifted = run(orc, p, contract=False, tau=tau, bias=bias + np.array([[0.3], [-1.1]]))
    np.testing.assert_allclose(shifted["loss_tok"], out["loss_tok"], rtol=0, atol=1e-12)
    np.testing.assert_allclose(shifted["dtau"], out["dtau"], rtol=1e-10, atol=1e-14)
    for k in range(p["K"]):
        assert rel(shifted["dhidden"][k], out["dhidden"][k]) < 1e-10


def pin_heads_torch_fp64(orc):
    """tau and b as autograd leaves of F.rms_norm, matmul and F.cross_entropy."""
    import torch
    import torch.nn.functional as F
    p = problem(K=3, N=7, d=16, V=30, seed=31, mask_frac=0.2, row_scale=True, orc=orc)
    p["W"] = p["W"] * 5.0
    tau, bias = _heads(p, 3)
    out = run(orc, p, contract=False, tau=tau, bias=bias)
    W = torch.tensor(p["W"], dtype=torch.float64, requires_grad=True)
    g = torch.tensor(p["gamma"], dtype=torch.float64, requires_grad=True)
    for k in range(p["K"]):
        t = torch.tensor(tau[k], dtype=torch.float64, requires_grad=True)
        b = torch.tensor(bias[k], dtype=torch.float64, requires_grad=True)
        h = torch.tensor(p["hidden"][k], dtype=torch.float64, requires_grad=True)
        y = torch.tensor(p["targets"][k], dtype=torch.int64)
        x = F.rms_norm(h, (p["d"],), weight=g, eps=p["eps"])
        loss = F.cross_entropy(t * (x @ W.T) + b, y, ignore_index=-100)
        W.grad = None
        g.grad = None
        loss.backward()
        assert abs(loss.item() - out["loss_mean"][k]) < 1e-12
        assert abs(t.grad.item() - out["dtau"][k]) < 1e-12 * max(1.0, abs(t.grad.item()))
        assert rel(out["dbias"][k], b.grad.numpy()) < 1e-11
        assert rel(out["dhidden"][k], h.grad.numpy()) < 1e-11
        if k == p["K"] - 1:
            assert rel(out["dW"], W.grad.numpy()) < 1e-11
            assert rel(out["dgamma"], g.grad.numpy()) < 1e-11


PINS += [pin_heads_finite_differences, pin_heads_closed_forms, pin_heads_torch_fp64]


# -- private readouts -----------------------------------------------------------

def pin_private_readouts(orc):
    """With every W_k = W and gamma_k = gamma the private readouts reduce to the
    shared one (losses, dH, and the final module's dW, dgamma); a module's own
    dW_k and dgamma_k match central differences of its own loss."""
    p = problem(K=3, N=5, d=8, V=12, seed=33, mask_frac=0.2, row_scale=True, orc=orc)
    p["W"] = p["W"] * 15.0
    K = p["K"]
    shared = run(orc, p, contract=True)
    priv = orc.solo_readout_private(p["hidden"], [p["gamma"]] * K, [p["W"]] * K, p["targets"],
                                    eps=p["eps"], contract=True)
    np.testing.assert_allclose(priv["loss_tok"], shared["loss_tok"], rtol=0, atol=1e-14)
    for k in range(K):
        assert rel(priv["dhidden"][k], shared["dhidden"][k]) < 1e-13
    assert rel(priv["dW"][-1], shared["dW"]) < 1e-13
    assert rel(priv["dgamma"][-1], shared["dgamma"]) < 1e-13
    # distinct readouts: FD of module 0's loss in its own W_0 and gamma_0
    rng = np.random.default_rng(4)
    Ws = [p["W"] * (1.0 + 0.3 * rng.standard_normal(p["W"].shape)) for _ in range(K)]
    gs = [p["gamma"] * (1.0 + 0.2 * rng.standard_normal(p["d"])) for _ in range(K)]
    out = orc.solo_readout_private(p["hidden"], gs, Ws, p["targets"], eps=p["eps"],
                                   contract=False)
    step = 1e-6
    L0 = lambda W0, g0: orc.solo_readout_private(p["hidden"][:1], [g0], [W0], p["targets"][:1],
                                                 eps=p["eps"], contract=False)["loss_mean"][0]
    numW = np.zeros_like(Ws[0])
    for idx in np.ndindex(*numW.shape):
        Wp, Wm = Ws[0].copy(), Ws[0].copy()
        Wp[idx] += step
        Wm[idx] -= step
        numW[idx] = (L0(Wp, gs[0]) - L0(Wm, gs[0])) / (2 * step)
    assert rel(out["dW"][0], numW) < 1e-7
    numg = np.zeros(p["d"])
    for j in range(p["d"]):
        gp, gm = gs[0].copy(), gs[0].copy()
        gp[j] += step
        gm[j] -= step
        numg[j] = (L0(Ws[0], gp) - L0(Ws[0], gm)) / (2 * step)
    assert rel(out["dgamma"][0], numg) < 1e-7


PINS.append(pin_private_readouts)
