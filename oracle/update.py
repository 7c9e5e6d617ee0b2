"""Oracle drafter-head update (Sec. 3.4; test infrastructure only).

For N logged tuples with head inputs U [N, d] (u = RMSNorm_final(h_k)),
drafted tokens a, verifier logits l = logits^phi, verifier argmax y* and
rewards r (1 accepted, 0 first reject):

  drafter logits   Z = U (W^(S) + gamma A B)^T           p = softmax(Z)
  teacher          q_tau = softmax(l / tau),  q_1 = softmax(l)

  L_fast   = lambda_kl * mean_all KL(p || q_tau)
           + lambda_pg * L_pg,   L_pg = -(1/|P|) sum_{P} log p(a)   (P: r = 1)
           + w_ce * mean_all [-log p(y*)]
           - w_ent * mean_all H[p]
  L_policy = w_rl * mean_{accepted and first reject} [-(r - b) log p(a)]
           + beta(t) * mean_all KL(p || q_1)
  L        = L_fast + [t >= T_warmup] L_policy      ("dvi" objective)

The KL->RL schedule is the piecewise-linear (lambda_pg, lambda_kl)(t) of
Sec. 3.4 over completed updates t.  The paper leaves L_CE, the row sets of the
KL and entropy terms, beta(t), w_rl(t), the baseline's EMA constant and the
optimizer unnamed; the readings used here: L_CE is the hard CE to the
verifier's y*, KL/entropy/CE use every logged row, beta(t) decays
exponentially from beta0 to beta_min after warmup, w_rl ramps like lambda_pg,
b is an EMA (rho) of the rewards updated after the loss is formed, and the
optimizer is bias-corrected Adam.  A mean over an empty set is 0.

Gradient with respect to one row z of Z (p = softmax(z)):
  d KL(p||q)/dz_j   = p_j (log p_j - log q_j - KL)
  d (-log p_a)/dz_j = p_j - [j = a]
  d (-H)/dz_j       = p_j (log p_j + H)
and with G = dL/dZ:  dA = gamma G^T (U B^T),  dB = gamma (G A)^T U,
dW^(S) = G^T U (full-head mode).
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import List, Optional

import numpy as np

from .model import log_softmax, OracleModel


@dataclass(frozen=True)
class ObjectiveWeights:
    lam_kl: float
    lam_pg: float
    w_ce: float
    w_ent: float
    w_rl: float
    beta: float
    tau: float


def kl_rl_schedule(t: int, h):
    """(lambda_pg, lambda_kl) at update t: warmup, linear ramp, then flat (Sec. 3.4)."""
    if t < h.t_warmup:
        return 0.0, h.lambda0
    if t < h.t_warmup + h.t_ramp:
        f = (t - h.t_warmup) / h.t_ramp
        return f * h.lambda_pg_max, h.lambda0 - f * (h.lambda0 - h.lambda_kl_min)
    return h.lambda_pg_max, h.lambda_kl_min


def objective_weights(t: int, h) -> ObjectiveWeights:
    """Weights of every loss term at update t for the chosen objective.

    "dvi": the KL->RL schedule plus L_policy from T_warmup on.  The single-term
    ablations of Sec. 4.3: "kl" (online distillation), "pg" (REINFORCE),
    "ce" (reward-masked cross-entropy).
    """
    if h.objective == "kl":
        return ObjectiveWeights(h.lambda0, 0.0, 0.0, 0.0, 0.0, 0.0, h.tau)
    if h.objective == "pg":
        return ObjectiveWeights(0.0, 0.0, 0.0, 0.0, 1.0, 0.0, h.tau)
    if h.objective == "ce":
        return ObjectiveWeights(0.0, 1.0, 0.0, 0.0, 0.0, 0.0, h.tau)
    lam_pg, lam_kl = kl_rl_schedule(t, h)
    if t >= h.t_warmup:
        frac = min(1.0, (t - h.t_warmup) / h.t_ramp) if h.t_ramp > 0 else 1.0
        w_rl = h.w_rl_max * frac
        beta = h.beta_min + (h.beta0 - h.beta_min) * np.exp(-(t - h.t_warmup) / h.t_beta)
    else:
        w_rl, beta = 0.0, 0.0
    return ObjectiveWeights(lam_kl, lam_pg, h.w_ce, h.w_ent, w_rl, float(beta), h.tau)


def head_logits(U, W_s, A, B, gamma):
    """Z = U W_s^T + gamma (U B^T) A^T, i.e. the drafter head (W^S + gamma A B) u."""
    Z = U @ W_s.T
    if A is not None and A.shape[1] > 0:
        Z = Z + gamma * (U @ B.T) @ A.T
    return Z


def loss_terms(Z, logits_phi, a, ystar, tau):
    """Per-row pieces: log p, p, KL(p||q_tau), KL(p||q_1), H[p], -log p(a), -log p(y*)."""
    lp = log_softmax(Z)
    p = np.exp(lp)
    lq = log_softmax(logits_phi / tau)
    lq1 = log_softmax(logits_phi)
    rows = np.arange(Z.shape[0])
    return dict(
        lp=lp, p=p, lq=lq, lq1=lq1,
        kl=np.sum(p * (lp - lq), axis=1),
        kl1=np.sum(p * (lp - lq1), axis=1),
        ent=-np.sum(p * lp, axis=1),
        nll_a=-lp[rows, a],
        nll_y=-lp[rows, ystar],
    )


def _mean(x, mask=None):
    if mask is not None:
        x = x[mask]
    return float(np.mean(x)) if x.size else 0.0


def total_loss(Z, logits_phi, a, ystar, r, w: ObjectiveWeights, b: float):
    """Scalar objective L and its named parts (means over the logged rows)."""
    t = loss_terms(Z, logits_phi, a, ystar, w.tau)
    acc = r == 1
    parts = dict(
        kl=_mean(t["kl"]), pg=_mean(t["nll_a"], acc), ce=_mean(t["nll_y"]),
        ent=_mean(t["ent"]), rl=_mean((r - b) * t["nll_a"]), kl1=_mean(t["kl1"]))
    L = (w.lam_kl * parts["kl"] + w.lam_pg * parts["pg"] + w.w_ce * parts["ce"]
         - w.w_ent * parts["ent"] + w.w_rl * parts["rl"] + w.beta * parts["kl1"])
    return L, parts


def grad_logits(Z, logits_phi, a, ystar, r, w: ObjectiveWeights, b: float):
    """G = dL/dZ, row by row from the closed forms in the module docstring."""
    t = loss_terms(Z, logits_phi, a, ystar, w.tau)
    N, V = Z.shape
    p, lp = t["p"], t["lp"]
    acc = (r == 1)
    nP = int(acc.sum())
    G = (w.lam_kl / N) * p * (lp - t["lq"] - t["kl"][:, None])
    G = G + (w.beta / N) * p * (lp - t["lq1"] - t["kl1"][:, None])
    G = G + (w.w_ent / N) * p * (lp + t["ent"][:, None])
    ca = (w.lam_pg * acc / nP if nP else np.zeros(N)) + w.w_rl * (r - b) / N
    onehot_a = np.zeros_like(p)
    onehot_a[np.arange(N), a] = 1.0
    onehot_y = np.zeros_like(p)
    onehot_y[np.arange(N), ystar] = 1.0
    G = G + ca[:, None] * (p - onehot_a) + (w.w_ce / N) * (p - onehot_y)
    return G


def param_grads(G, U, A, B, gamma, full: bool = False):
    """Chain rule through Z = U W_s^T + gamma (U B^T) A^T."""
    if full:
        return {"W_s": G.T @ U}
    UB = U @ B.T
    return {"A": gamma * G.T @ UB, "B": gamma * (G @ A).T @ U}


@dataclass
class AdamState:
    m: np.ndarray
    v: np.ndarray
    step: int = 0


def adam_step(param, grad, st: AdamState, lr, b1, b2, eps):
    """Bias-corrected Adam, in place on `param`."""
    st.step += 1
    st.m[...] = b1 * st.m + (1.0 - b1) * grad
    st.v[...] = b2 * st.v + (1.0 - b2) * grad * grad
    mhat = st.m / (1.0 - b1 ** st.step)
    vhat = st.v / (1.0 - b2 ** st.step)
    param -= lr * mhat / (np.sqrt(vhat) + eps)


class DrafterUpdater:
    """Owns theta (A, B, or W^S in full-head mode), optimizer state, t and b."""

    def __init__(self, model: OracleModel, hyper, full: bool = False):
        self.model, self.h, self.full = model, hyper, full
        self.t = 0
        self.b = 0.0
        names = ["w_s"] if full else ["lora_a", "lora_b"]
        self.params = names
        self.opt = {n: AdamState(np.zeros_like(getattr(model, n)),
                                 np.zeros_like(getattr(model, n))) for n in names}

    def update(self, tuples) -> dict:
        md, h = self.model, self.h
        info = dict(t=self.t, n=len(tuples), b_before=self.b)
        w = objective_weights(self.t, h)
        info["weights"] = w
        if not tuples:
            self.t += 1
            info.update(loss=0.0, skipped=True)
            return info
        U = np.stack([x.u for x in tuples]).astype(md.dtype)
        Lg = np.stack([x.logits for x in tuples]).astype(md.dtype)
        a = np.array([x.a for x in tuples])
        ys = np.array([x.ystar for x in tuples])
        r = np.array([x.r for x in tuples], dtype=md.dtype)
        Z = head_logits(U, md.w_s, md.lora_a, md.lora_b, md.gamma)
        L, parts = total_loss(Z, Lg, a, ys, r, w, self.b)
        info.update(loss=L, parts=parts, accept_rate=float(np.mean(r)))
        if not np.isfinite(L):
            info["skipped"] = True
            self.t += 1
            return info
        G = grad_logits(Z, Lg, a, ys, r, w, self.b)
        grads = param_grads(G, U, md.lora_a, md.lora_b, md.gamma, self.full)
        info["grads"] = {("W_s" if k == "W_s" else k): v.copy() for k, v in grads.items()}
        for name in self.params:
            g = grads["W_s" if name == "w_s" else ("A" if name == "lora_a" else "B")]
            P = getattr(md, name)
            if h.optimizer == "sgd":
                P -= h.lr * g
            else:
                adam_step(P, g, self.opt[name], h.lr, h.beta1, h.beta2, h.adam_eps)
        self.b = h.baseline_rho * self.b + (1.0 - h.baseline_rho) * float(np.mean(r))
        self.t += 1
        info["b_after"] = self.b
        return info
