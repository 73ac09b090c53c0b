"""Helpers of the GPU parity tests: upload seeded inputs, run the library,
run the oracle on the same bytes and compare with the stated tolerances.

Tolerances (per the headline specification of this path):
  per-token loss   abs err <= 2e-3
  module mean loss rel err <= 1e-4
  dH, dW, dgamma   max_abs(gpu - oracle) / max_abs(oracle) <= 2e-2, and
                   cosine similarity >= 0.9999
The oracle runs in "contract" mode: xhat is rounded to bf16 exactly where
the GPU rounds it; everything after is fp64.
"""
from __future__ import annotations

import numpy as np

import oracle.solo_oracle as orc
from paper_2609_35440_gb300 import synth

LOSS_TOK_ABS = 2e-3
LOSS_MEAN_REL = 1e-4
GRAD_REL = 2e-2
GRAD_COS = 0.9999


def to_device_bf16(bits: np.ndarray, device="cuda"):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16))
    return t.to(device).view(torch.bfloat16)


def bf16_tensor_to_f64(t) -> np.ndarray:
    import torch
    return orc.bf16_bits_to_f64(t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16))


def run_gpu(wl, inp: synth.Inputs, mask: np.ndarray | None = None, want_dW=True,
            want_dgamma=True, want_loss_tok=True, targets: np.ndarray | None = None,
            onchip: bool = False):
    import torch
    from paper_2609_35440_gb300 import solo_readout as sr
    dev = torch.device("cuda")
    hidden = [to_device_bf16(inp.hidden[k]) for k in range(wl.K)]
    gamma = to_device_bf16(inp.gamma)
    W = to_device_bf16(inp.W)
    tg = inp.targets if targets is None else targets
    tgt = torch.from_numpy(np.ascontiguousarray(tg, dtype=np.int32)).to(dev)
    mk = None if mask is None else torch.from_numpy(np.ascontiguousarray(mask, np.uint8)).to(dev)
    ro = sr.Readout(wl.K, wl.N, wl.d, wl.V, eps=wl.eps, ignore_index=wl.ignore_index,
                    want_loss_tok=want_loss_tok, want_dW=want_dW, want_dgamma=want_dgamma,
                    onchip=onchip)
    ro(hidden, gamma, W, tgt, mk)
    flags = ro.flags()
    torch.cuda.synchronize()
    out = dict(loss_mean=ro.loss_mean.double().cpu().numpy(), flags=flags,
               dhidden=[bf16_tensor_to_f64(x) for x in ro.dhidden])
    if want_loss_tok:
        out["loss_tok"] = ro.loss_tok.double().cpu().numpy()
    if want_dW:
        out["dW"] = ro.dW.double().cpu().numpy()
    if want_dgamma:
        out["dgamma"] = ro.dgamma.double().cpu().numpy()
    out["_ro"] = ro
    return out


def oracle_full(wl, inp: synth.Inputs, mask=None, targets=None):
    dec = orc.bf16_bits_to_f64
    hidden = [dec(inp.hidden[k]) for k in range(wl.K)]
    tg = inp.targets if targets is None else targets
    # the library receives eps as fp32; the oracle uses that same value
    return orc.solo_readout_fwd_bwd(hidden, dec(inp.gamma), dec(inp.W), tg.astype(np.int64),
                                    mask, eps=float(np.float32(wl.eps)),
                                    ignore_index=wl.ignore_index, contract=True)


def max_rel(a, ref) -> float:
    a, ref = np.asarray(a, np.float64), np.asarray(ref, np.float64)
    den = np.max(np.abs(ref)) if ref.size else 0.0
    num = np.max(np.abs(a - ref)) if ref.size else 0.0
    if den == 0.0:
        return float(num)
    return float(num / den)


def cosine(a, ref) -> float:
    a, ref = np.ravel(np.asarray(a, np.float64)), np.ravel(np.asarray(ref, np.float64))
    na, nr = np.linalg.norm(a), np.linalg.norm(ref)
    if na == 0.0 and nr == 0.0:
        return 1.0
    return float(np.dot(a, ref) / (na * nr))


def check_grad(name, a, ref, report):
    mr, cs = max_rel(a, ref), cosine(a, ref)
    report[name] = (mr, cs)
    zero_ref = not np.any(ref)
    if zero_ref:
        assert np.max(np.abs(a)) <= 1e-6, (name, "reference is zero", np.max(np.abs(a)))
        return
    assert mr <= GRAD_REL, (name, "max rel err", mr)
    assert cs >= GRAD_COS, (name, "cosine", cs)


def compare_full(wl, gpu, ref, check_dW=True, check_dgamma=True):
    """Element-by-element comparison of every output; returns the error report."""
    rep = {}
    lt_err = float(np.max(np.abs(gpu["loss_tok"] - ref["loss_tok"])))
    rep["loss_tok_abs"] = lt_err
    assert lt_err <= LOSS_TOK_ABS, ("loss_tok", lt_err)
    for k in range(wl.K):
        want = ref["loss_mean"][k]
        got = gpu["loss_mean"][k]
        if want == 0.0:
            assert got == 0.0, ("loss_mean", k, got)
        else:
            assert abs(got - want) / abs(want) <= LOSS_MEAN_REL, ("loss_mean", k, got, want)
        check_grad(f"dH[{k}]", gpu["dhidden"][k], ref["dhidden"][k], rep)
    if check_dW:
        check_grad("dW", gpu["dW"], ref["dW"], rep)
    if check_dgamma:
        check_grad("dgamma", gpu["dgamma"], ref["dgamma"], rep)
    return rep


def sampled_check(wl, inp: synth.Inputs, gpu, rows_per_module=24, n_vocab=48, seed=0,
                  full_final=True, chunk=512):
    """Parity at full size on sampled outputs the oracle computes one by one.

    For every module: the first and last token and random tokens: token loss
    (abs err) and dH rows (max rel err and cosine over the sampled rows).  The
    module mean must equal the mean of the kept token losses (a property).
    With ``full_final`` the final module is run through the oracle in chunks:
    its mean loss, every dgamma entry and the dW rows of sampled vocabulary
    entries (including heavy rows and frequent targets) are compared.
    """
    rng = np.random.default_rng(seed)
    dec = orc.bf16_bits_to_f64
    gamma, W = dec(inp.gamma), dec(inp.W)
    eps = float(np.float32(wl.eps))
    rep = {}
    for k in range(wl.K):
        y = inp.targets[k].astype(np.int64)
        kept, _ = orc.kept_tokens(y, None, wl.V, wl.ignore_index)
        nv = int(kept.sum())
        rows = np.unique(np.concatenate([[0, wl.N - 1],
                                         rng.choice(wl.N, min(rows_per_module, wl.N), replace=False)]))
        res = orc.module_rows(dec(inp.hidden[k][rows]), gamma, W, y[rows], kept[rows], nv, eps, True)
        err = float(np.max(np.abs(gpu["loss_tok"][k][rows] - res["loss"])))
        rep[f"loss_tok[{k}]"] = err
        assert err <= LOSS_TOK_ABS, ("loss_tok", k, err)
        check_grad(f"dH[{k}] rows", gpu["dhidden"][k][rows], res["dh"], rep)
        mean_prop = float(np.sum(gpu["loss_tok"][k][kept], dtype=np.float64) / max(nv, 1))
        assert abs(gpu["loss_mean"][k] - mean_prop) <= 1e-6 * max(1.0, abs(mean_prop)), \
            ("loss_mean property", k, gpu["loss_mean"][k], mean_prop)
    if full_final:
        k = wl.K - 1
        y = inp.targets[k].astype(np.int64)
        kept, _ = orc.kept_tokens(y, None, wl.V, wl.ignore_index)
        Wrms = np.sqrt(np.mean(W * W, axis=1))
        heavy = np.nonzero(Wrms > 5 * np.median(Wrms))[0][:8]
        freq = np.argsort(-np.bincount(y[kept], minlength=wl.V))[:8]
        cols = np.unique(np.concatenate([[0, wl.V - 1], heavy, freq,
                                         rng.choice(wl.V, n_vocab, replace=False)]))
        ch = orc.final_module_chunked(lambda i0, n: dec(inp.hidden[k][i0:i0 + n]), wl.N, gamma,
                                      W, y, kept, eps, True, dW_cols=cols, chunk=chunk)
        want = ch["loss"].sum() / max(ch["n_valid"], 1)
        rel = abs(gpu["loss_mean"][k] - want) / abs(want)
        rep["loss_mean_final_rel"] = rel
        assert rel <= LOSS_MEAN_REL, ("loss_mean", k, gpu["loss_mean"][k], want)
        # every token loss of the final module, element by element
        err = float(np.max(np.abs(gpu["loss_tok"][k] - ch["loss"])))
        rep["loss_tok_final_all"] = err
        assert err <= LOSS_TOK_ABS, ("loss_tok of the final module", err)
        check_grad("dgamma", gpu["dgamma"], ch["dgamma"], rep)
        check_grad("dW rows", gpu["dW"][cols], ch["dW_rows"], rep)
    # each column of dW sums to zero over the vocabulary (rows of G sum to zero)
    colsum = np.abs(gpu["dW"].sum(axis=0))
    scale = np.sqrt(np.sum(gpu["dW"] ** 2, axis=0)) + 1e-30
    rep["dW_colsum_rel"] = float(np.max(colsum / scale))
    assert rep["dW_colsum_rel"] < 1e-2, rep["dW_colsum_rel"]
    return rep
