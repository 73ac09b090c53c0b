"""Plants plausible mistakes in copies of the oracle (CPU only) and checks
that at least one pin catches each: a pin set that cannot see a dropped
term, a wrong sign, a wrong index or a transposed operand pins nothing."""
import importlib.util

import numpy as np
import pytest

from tests.oracle_pins import PINS


def fresh_oracle():
    spec = importlib.util.find_spec("oracle.solo_oracle")
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _mut_rms_bwd_drop_term(o):
    o.rmsnorm_backward = lambda dx, h, g, r: r[:, None] * g[None, :] * dx


def _mut_rms_bwd_sign(o):
    def f(dx, h, g, r):
        d = h.shape[1]
        c = np.sum(g[None, :] * dx * h, axis=1)
        return r[:, None] * g[None, :] * dx + (r ** 3 / d)[:, None] * h * c[:, None]
    o.rmsnorm_backward = f


def _mut_rms_bwd_power(o):
    def f(dx, h, g, r):
        d = h.shape[1]
        c = np.sum(g[None, :] * dx * h, axis=1)
        return r[:, None] * g[None, :] * dx - (r ** 2 / d)[:, None] * h * c[:, None]
    o.rmsnorm_backward = f


def _mut_rms_fwd_eps_outside(o):
    def f(h, g, eps, contract=True):
        r = 1.0 / (np.sqrt(np.mean(h * h, axis=1)) + eps)
        x = g[None, :] * h * r[:, None]
        return r, (o.round_to_bf16(x) if contract else x)
    o.rmsnorm_forward = f


def _mut_rms_fwd_no_gain(o):
    def f(h, g, eps, contract=True):
        r = 1.0 / np.sqrt(np.mean(h * h, axis=1) + eps)
        x = h * r[:, None]
        return r, (o.round_to_bf16(x) if contract else x)
    o.rmsnorm_forward = f


def _mut_rms_fwd_sum_not_mean(o):
    def f(h, g, eps, contract=True):
        r = 1.0 / np.sqrt(np.sum(h * h, axis=1) + eps)
        x = g[None, :] * h * r[:, None]
        return r, (o.round_to_bf16(x) if contract else x)
    o.rmsnorm_forward = f


def _mut_grad_no_onehot(o):
    def f(z, lse, y, kept, n_valid):
        g = np.exp(z - lse[:, None])
        return g * np.where(kept, 1.0 / max(n_valid, 1), 0.0)[:, None]
    o.logit_grad = f


def _mut_grad_mean_over_all(o):
    def f(z, lse, y, kept, n_valid):
        g = np.exp(z - lse[:, None])
        rows = np.nonzero(kept)[0]
        g[rows, y[rows]] -= 1.0
        return g * np.where(kept, 1.0 / len(y), 0.0)[:, None]
    o.logit_grad = f


def _mut_grad_onehot_wrong_index(o):
    def f(z, lse, y, kept, n_valid):
        g = np.exp(z - lse[:, None])
        rows = np.nonzero(kept)[0]
        g[rows, (y[rows] + 1) % z.shape[1]] -= 1.0
        return g * np.where(kept, 1.0 / max(n_valid, 1), 0.0)[:, None]
    o.logit_grad = f


def _mut_lse_drop_max(o):
    o.log_sum_exp = lambda z: np.log(np.sum(np.exp(z - np.max(z, axis=1)[:, None]), axis=1))


def _mut_loss_sign(o):
    def f(z, lse, y, kept):
        rows = np.arange(z.shape[0])
        return np.where(kept, z[rows, np.where(kept, y, 0)] - lse, 0.0)
    o.token_loss = f


def _mut_logits_reversed_width(o):
    o.logits = lambda x, W: x[:, ::-1] @ W.T


def _mut_logits_transposed(o):
    o.logits = lambda x, W: (W @ x.T).T if W.shape[0] == x.shape[1] else x @ W[:, :x.shape[1]].T[:, ::-1]


def _mut_input_grad_reversed(o):
    o.input_grad = lambda g, W: g @ W[:, ::-1]


def _mut_dW_no_onehot_rows(o):
    def f(g, xhat, dxhat, h, r):
        return g.T @ xhat[::-1], np.sum(dxhat * h * r[:, None], axis=0)
    o.readout_grads = f


def _mut_dgamma_no_r(o):
    def f(g, xhat, dxhat, h, r):
        return g.T @ xhat, np.sum(dxhat * h, axis=0)
    o.readout_grads = f


def _mut_round_half_up(o):
    def q(x):
        m, e = np.frexp(np.asarray(x, dtype=np.float64))
        return np.ldexp(np.floor(m * 256.0 + 0.5) / 256.0, e)
    o.round_to_bf16 = q


def _mut_round_truncate(o):
    def q(x):
        m, e = np.frexp(np.asarray(x, dtype=np.float64))
        return np.ldexp(np.trunc(m * 256.0) / 256.0, e)
    o.round_to_bf16 = q


def _mut_kept_ignores_mask(o):
    orig = o.kept_tokens
    o.kept_tokens = lambda t, mask, V, ii: orig(t, None, V, ii)


def _mut_bad_target_not_masked(o):
    def f(t, mask, V, ii):
        t = np.asarray(t)
        kept = (t != ii) & (t >= 0)
        if mask is not None:
            kept &= np.asarray(mask) != 0
        return kept & (t < V + 1), np.zeros_like(kept)
    o.kept_tokens = f


def _mut_exit_last_argmax(o):
    orig = o.exit_readout

    def f(*a, **kw):
        out = orig(*a, **kw)
        out["top1"] = np.stack([z.shape[1] - 1 - np.argmax(z[:, ::-1], axis=1) for z in out["z"]])
        return out
    o.exit_readout = f


def _mut_exit_logprob_without_lse(o):
    orig = o.exit_readout

    def f(*a, **kw):
        out = orig(*a, **kw)
        out["top1_logprob"] = np.stack([np.max(z, axis=1) for z in out["z"]])
        return out
    o.exit_readout = f


def _mut_heads_tau_missing_in_dh(o):
    orig = o.module_rows

    def f(h, gamma, W, y, kept, n_valid, eps, contract=True, tau=1.0, b=None):
        res = orig(h, gamma, W, y, kept, n_valid, eps, contract, tau, b)
        res["dxhat"] = o.input_grad(res["g"], W)
        res["dh"] = o.rmsnorm_backward(res["dxhat"], h, gamma, res["r"])
        return res
    o.module_rows = f


def _mut_heads_dtau_uses_z(o):
    orig = o.module_rows

    def f(h, gamma, W, y, kept, n_valid, eps, contract=True, tau=1.0, b=None):
        res = orig(h, gamma, W, y, kept, n_valid, eps, contract, tau, b)
        res["dtau"] = float(np.sum(res["g"] * res["z"]))
        return res
    o.module_rows = f


def _mut_heads_db_times_tau(o):
    orig = o.module_rows

    def f(h, gamma, W, y, kept, n_valid, eps, contract=True, tau=1.0, b=None):
        res = orig(h, gamma, W, y, kept, n_valid, eps, contract, tau, b)
        res["db"] = tau * res["db"]
        return res
    o.module_rows = f


def _mut_heads_bias_scaled_by_tau(o):
    o.head_logits = lambda s, tau=1.0, b=None: tau * (s if b is None else s + b[None, :])


MUTATIONS = [v for k, v in sorted(globals().items()) if k.startswith("_mut_")]


@pytest.mark.parametrize("mut", MUTATIONS, ids=[m.__name__[5:] for m in MUTATIONS])
def test_planted_mistake_is_caught(mut):
    o = fresh_oracle()
    mut(o)
    caught = []
    for pin in PINS:
        try:
            with np.errstate(all="ignore"):
                pin(o)
        except Exception as e:  # AssertionError, or a shape error from a wrong operand
            caught.append((pin.__name__, type(e).__name__))
    assert caught, f"no pin catches mutation {mut.__name__}"
