"""Float64 restatements of the paper's two reductions to attention.

These are independent algebraic routes to the Gauss sum, used only to pin
the oracle (they share no code with it):

* Alg. 1 (prescale): v~_n = v_n exp(-tau/2 ||k_n||^2), then softmax
  attention with its log-sum-exp, then s_m = Att_m exp(lse_m) exp(-tau/2 ||q_m||^2).
* Alg. 2 (reweight): q~ = [q, 1, ||q||^2/2], k~ = [k, -||k||^2/2, 0] plus the
  extra key k~_0 = e_{D+2} with value kappa e_{C+1}, kappa = sqrt(N+1);
  [alpha, beta] = Att(q~, k~, v~); s = kappa alpha / beta.

Softmax attention (Eq. 2) is evaluated in the usual stable way, subtracting
the row maximum of the logits.
"""
import numpy as np


def attention(q, k, v, tau):
    """Att_tau(q, k, v) and lse_tau(q, k) of Eq. 2, float64."""
    logits = tau * (q @ k.T)
    mx = logits.max(axis=1, keepdims=True)
    w = np.exp(logits - mx)
    den = w.sum(axis=1, keepdims=True)
    att = (w @ v) / den
    lse = (mx + np.log(den))[:, 0]
    return att, lse


def prescale(q, k, v, tau):
    """Alg. 1."""
    vt = v * np.exp(-0.5 * tau * np.sum(k * k, axis=1))[:, None]
    att, lse = attention(q, k, vt, tau)
    return att * np.exp(lse - 0.5 * tau * np.sum(q * q, axis=1))[:, None]


def reweight(q, k, v, tau, return_parts=False):
    """Alg. 2 (and, on request, alpha, beta and kappa for Prop. 1)."""
    M, D = q.shape
    N, C = v.shape
    kappa = np.sqrt(N + 1.0)
    qt = np.concatenate([q, np.ones((M, 1)), 0.5 * np.sum(q * q, axis=1, keepdims=True)], axis=1)
    kt = np.concatenate([k, -0.5 * np.sum(k * k, axis=1, keepdims=True), np.zeros((N, 1))], axis=1)
    k0 = np.zeros((1, D + 2))
    k0[0, D + 1] = 1.0
    kt = np.concatenate([k0, kt], axis=0)
    vt = np.concatenate([v, np.zeros((N, 1))], axis=1)
    v0 = np.zeros((1, C + 1))
    v0[0, C] = kappa
    vt = np.concatenate([v0, vt], axis=0)
    att, _ = attention(qt, kt, vt, tau)
    alpha, beta = att[:, :C], att[:, C]
    s = kappa * alpha / beta[:, None]
    if return_parts:
        return s, alpha, beta, kappa
    return s
