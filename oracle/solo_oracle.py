"""fp64 CPU oracle of the SOLO shared-readout local loss.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this module.  It shares no
code with the CUDA library and never calls it.

What it computes, for every module k and token i (paper, Section 2.2, Eq. 2
with tau_k = 1 and no bias; Eq. 3; Algorithm 1, the local cross-entropy of
each module and the terminal cross-entropy that updates W; the head's final
RMSNorm with element-wise gain, Appendix C "Language" and the ROT/RSHARE
paragraph of Appendix D):

1. ms_i = (1/d) sum_j h_ij^2,   r_i = 1 / sqrt(ms_i + eps)
2. xhat_ij = Q(gamma_j h_ij r_i)        Q = bf16 round-to-nearest-even in
                                         "contract" mode, identity in "exact"
3. z_iv = sum_j xhat_ij W_vj             (logits through the shared readout)
4. lse_i = max_v z + ln sum_v exp(z_iv - max_v z)
   loss_i = lse_i - z_{i,y_i} for kept tokens, 0 otherwise
   L_k = sum_i loss_i / Nvalid_k (0 when no token is kept)
5. g_iv = (exp(z_iv - lse_i) - [v = y_i]) / Nvalid_k   (delta_k of Eq. 1,
   scaled by the mean; zero rows for masked tokens)
6. dxhat = g W                            (the readout factor W^T delta_k, Eq. 3)
7. dh_ij = r_i gamma_j dxhat_ij - (r_i^3/d) h_ij sum_l gamma_l dxhat_il h_il
   (Jacobian of the final RMSNorm)
8. final module only (Algorithm 1: only the terminal loss updates W):
   dW_vj = sum_i g_iv xhat_ij,   dgamma_j = sum_i dxhat_ij h_ij r_i

With the heads' own parameters (Algorithm 1: the local loss of module k is
CE(softmax(tau_k W-bar phi_k(h_k) + b_k), y), the terminal CE(W h_K + b, y))
step 3 becomes z = tau_k s + b_k with s = xhat W^T, the chain rule puts tau_k
in front of g in steps 6 and 8, and
9. dtau_k = sum_i sum_v g_iv s_iv,   db_k = sum_i g_i   (per module).

A token is kept when its target lies in [0, V), differs from ignore_index
and its optional mask byte is non-zero.  A target outside [0, V) that is not
ignore_index is treated as masked and reported (``bad_target``).

Every step is a plain numpy fp64 expression; the matrix products are the
only library primitive used.  Rows are independent given Nvalid_k, so
``module_rows`` may be called on any subset of a module's rows.
"""
from __future__ import annotations

import numpy as np


# -- inputs -----------------------------------------------------------------

def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) to exact float64 values."""
    u = np.asarray(bits).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Rounds float64 values to the nearest bf16 value, ties to even.

    bf16 keeps 8 significant bits.  With x = m * 2^e, 0.5 <= |m| < 1, the
    rounded value is rint(256 m) / 256 * 2^e (rint rounds half to even).
    Rounding happens once, from float64.  bf16 subnormals (|x| < 2^-126) are
    out of this oracle's range.
    """
    m, e = np.frexp(np.asarray(x, dtype=np.float64))
    return np.ldexp(np.rint(m * 256.0) / 256.0, e)


def kept_tokens(targets: np.ndarray, mask, V: int, ignore_index: int):
    """(kept, bad): kept tokens and targets that are neither valid nor ignore_index."""
    t = np.asarray(targets)
    in_range = (t >= 0) & (t < V)
    bad = (~in_range) & (t != ignore_index)
    kept = in_range & (t != ignore_index)
    if mask is not None:
        kept &= np.asarray(mask) != 0
    return kept, bad


# -- steps 1-2: final RMSNorm with gain --------------------------------------

def rmsnorm_forward(h, gamma, eps, contract=True):
    d = h.shape[1]
    ms = np.sum(h * h, axis=1) / d
    r = 1.0 / np.sqrt(ms + eps)
    xhat = gamma[None, :] * h * r[:, None]
    if contract:
        xhat = round_to_bf16(xhat)
    return r, xhat


# -- steps 3-5: logits, cross-entropy, its gradient ---------------------------

def logits(xhat, W):
    return xhat @ W.T


def log_sum_exp(z):
    m = np.max(z, axis=1)
    return m + np.log(np.sum(np.exp(z - m[:, None]), axis=1))


def token_loss(z, lse, y, kept):
    rows = np.arange(z.shape[0])
    yc = np.where(kept, y, 0)
    return np.where(kept, lse - z[rows, yc], 0.0)


def logit_grad(z, lse, y, kept, n_valid):
    """g = (softmax(z) - onehot(y)) / Nvalid on kept rows, 0 on the others."""
    g = np.exp(z - lse[:, None])
    rows = np.nonzero(kept)[0]
    g[rows, y[rows]] -= 1.0
    w = np.where(kept, 1.0 / max(n_valid, 1), 0.0)
    return g * w[:, None]


# -- steps 6-8: back through the readout and the norm -------------------------

def input_grad(g, W):
    return g @ W


def rmsnorm_backward(dxhat, h, gamma, r):
    d = h.shape[1]
    c = np.sum(gamma[None, :] * dxhat * h, axis=1)
    return (r[:, None] * gamma[None, :] * dxhat
            - (r ** 3 / d)[:, None] * h * c[:, None])


def readout_grads(g, xhat, dxhat, h, r, tau=1.0):
    """(dW, dgamma) summed over the given rows of the final module."""
    dW = tau * (g.T @ xhat)
    dgamma = np.sum(dxhat * h * r[:, None], axis=0)
    return dW, dgamma


# -- drivers ----------------------------------------------------------------

def head_logits(s, tau=1.0, b=None):
    """z = tau s + b: a head's temperature and bias on the shared readout's logits."""
    z = tau * s
    return z if b is None else z + b[None, :]


def module_rows(h, gamma, W, y, kept, n_valid, eps, contract=True, tau=1.0, b=None):
    """Every per-token quantity for a set of rows of one module."""
    r, xhat = rmsnorm_forward(h, gamma, eps, contract)
    s = logits(xhat, W)
    z = head_logits(s, tau, b)
    lse = log_sum_exp(z)
    loss = token_loss(z, lse, y, kept)
    g = logit_grad(z, lse, y, kept, n_valid)
    dxhat = tau * input_grad(g, W)
    dh = rmsnorm_backward(dxhat, h, gamma, r)
    zy = z[np.arange(len(y)), np.where(kept, y, 0)]
    dtau = float(np.sum(g * s))
    db = np.sum(g, axis=0)
    return dict(r=r, xhat=xhat, s=s, z=z, lse=lse, loss=loss, g=g, dxhat=dxhat,
                dh=dh, zy=zy, dtau=dtau, db=db, tau=tau)


def solo_readout_fwd_bwd(hidden, gamma, W, targets, mask=None, eps=1e-6,
                         ignore_index=-100, contract=True, want_dW=True,
                         want_dgamma=True, tau=None, bias=None):
    """Full oracle for small problems.

    hidden: sequence of K float64 arrays [N, d]; gamma [d]; W [V, d];
    targets int [K, N]; mask None or [K, N].  Returns a dict with loss_tok
    [K, N], loss_mean [K], n_valid [K], dhidden (list of [N, d]), dW [V, d]
    and dgamma [d] of the final module, bad_target (bool) and per-module
    intermediates ``rows`` (list of module_rows dicts).  With tau [K] and/or
    bias [K, V] (the heads' parameters) also dtau [K] and dbias [K, V].
    """
    K = len(hidden)
    V = W.shape[0]
    out = dict(loss_tok=[], loss_mean=np.zeros(K), n_valid=np.zeros(K, int),
               dhidden=[], rows=[], bad_target=False, dtau=np.zeros(K),
               dbias=np.zeros((K, V)))
    for k in range(K):
        kept, bad = kept_tokens(targets[k], None if mask is None else mask[k],
                                V, ignore_index)
        out["bad_target"] |= bool(bad.any())
        n_valid = int(kept.sum())
        tk = 1.0 if tau is None else float(tau[k])
        bk = None if bias is None else np.asarray(bias[k], dtype=np.float64)
        res = module_rows(hidden[k], gamma, W, np.asarray(targets[k]), kept,
                          n_valid, eps, contract, tau=tk, b=bk)
        out["dtau"][k] = res["dtau"]
        out["dbias"][k] = res["db"]
        out["loss_tok"].append(res["loss"])
        out["loss_mean"][k] = res["loss"].sum() / n_valid if n_valid else 0.0
        out["n_valid"][k] = n_valid
        out["dhidden"].append(res["dh"])
        out["rows"].append(res)
        if k == K - 1:
            dW, dgamma = readout_grads(res["g"], res["xhat"], res["dxhat"],
                                       hidden[k], res["r"], tau=tk)
            if want_dW:
                out["dW"] = dW
            if want_dgamma:
                out["dgamma"] = dgamma
    out["loss_tok"] = np.stack(out["loss_tok"])
    return out


def exit_readout(hidden, gamma, W, targets=None, mask=None, eps=1e-6, ignore_index=-100,
                 contract=True):
    """Decoding through the shared readout at every depth (the early exits of
    Section 3 and Appendix E): per token the first argmax of the logits and its
    log-probability, and with targets the token loss -log p(y) (0 when masked)
    and the mean over kept tokens of each module."""
    K = len(hidden)
    V = W.shape[0]
    out = dict(top1=[], top1_logprob=[], loss_tok=[], loss_mean=np.zeros(K), z=[])
    for k in range(K):
        r, xhat = rmsnorm_forward(hidden[k], gamma, eps, contract)
        z = logits(xhat, W)
        lse = log_sum_exp(z)
        top = np.argmax(z, axis=1)                 # first index among equal maxima
        rows = np.arange(z.shape[0])
        out["top1"].append(top)
        out["top1_logprob"].append(z[rows, top] - lse)
        out["z"].append(z)
        if targets is not None:
            kept, _ = kept_tokens(targets[k], None if mask is None else mask[k], V,
                                  ignore_index)
            y = np.asarray(targets[k])
            loss = token_loss(z, lse, y, kept)
            out["loss_tok"].append(loss)
            n_valid = int(kept.sum())
            out["loss_mean"][k] = loss.sum() / n_valid if n_valid else 0.0
    out["top1"] = np.stack(out["top1"])
    out["top1_logprob"] = np.stack(out["top1_logprob"])
    if targets is not None:
        out["loss_tok"] = np.stack(out["loss_tok"])
    return out


def solo_readout_private(hidden, gammas, Ws, targets, mask=None, eps=1e-6, ignore_index=-100,
                         contract=True, tau=None, bias=None):
    """Private readouts (the PRIV arm) with head-owned final norms: module k
    predicts through its own W_k and gain gamma_k and gets dW_k, dgamma_k; each
    module is the single-module problem of ``solo_readout_fwd_bwd``."""
    K = len(hidden)
    out = dict(loss_tok=[], loss_mean=np.zeros(K), dhidden=[], dW=[], dgamma=[],
               dtau=np.zeros(K), dbias=[], bad_target=False)
    for k in range(K):
        r = solo_readout_fwd_bwd([hidden[k]], gammas[k], Ws[k], targets[k:k + 1],
                                 None if mask is None else mask[k:k + 1], eps, ignore_index,
                                 contract, tau=None if tau is None else tau[k:k + 1],
                                 bias=None if bias is None else bias[k:k + 1])
        out["loss_tok"].append(r["loss_tok"][0])
        out["loss_mean"][k] = r["loss_mean"][0]
        out["dhidden"].append(r["dhidden"][0])
        out["dW"].append(r["dW"])
        out["dgamma"].append(r["dgamma"])
        out["dtau"][k] = r["dtau"][0]
        out["dbias"].append(r["dbias"][0])
        out["bad_target"] |= r["bad_target"]
    out["loss_tok"] = np.stack(out["loss_tok"])
    out["dbias"] = np.stack(out["dbias"])
    return out


def final_module_chunked(h_rows_fn, N, gamma, W, y, kept, eps, contract=True,
                         dW_cols=None, chunk=1024):
    """Final-module pass over all N rows in chunks, for full-size checks.

    ``h_rows_fn(i0, n)`` returns rows [i0, i0+n) of the module as float64.
    Returns loss [N], lse [N], dgamma [d], and dW rows ``dW_cols`` (the
    vocabulary entries v whose dW_v, an [len, d] array, is wanted).
    """
    n_valid = int(kept.sum())
    d = W.shape[1]
    loss = np.zeros(N)
    lse = np.zeros(N)
    dgamma = np.zeros(d)
    cols = None if dW_cols is None else np.asarray(dW_cols)
    dW_part = None if cols is None else np.zeros((len(cols), d))
    for i0 in range(0, N, chunk):
        n = min(chunk, N - i0)
        h = h_rows_fn(i0, n)
        res = module_rows(h, gamma, W, y[i0:i0 + n], kept[i0:i0 + n], n_valid,
                          eps, contract)
        loss[i0:i0 + n] = res["loss"]
        lse[i0:i0 + n] = res["lse"]
        dgamma += np.sum(res["dxhat"] * h * res["r"][:, None], axis=0)
        if cols is not None:
            dW_part += res["g"][:, cols].T @ res["xhat"]
    return dict(loss=loss, lse=lse, dgamma=dgamma, dW_rows=dW_part,
                n_valid=n_valid)
