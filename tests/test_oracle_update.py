"""Pins of the oracle's drafter update (Sec. 3.4).

* Every loss term's analytic gradient against central finite differences in
  fp64, through Z and through the parameters (LoRA A, B and full W^S).
* Closed forms: KL(p||p) = 0, uniform logits give CE = H = log V, two-class
  KL by hand, each gradient row sums to zero (softmax shift invariance).
* The KL->RL schedule at and around its breakpoints (continuity, end values,
  the linear midpoint).
* Adam's first two bias-corrected steps under a constant gradient move every
  coordinate by lr * sign(g); SGD moves by lr * g.
* Empty reward sets contribute nothing (no NaN); the baseline is an EMA.
"""
import dataclasses
import math

import numpy as np
import pytest

from oracle import (objective_weights, head_logits, total_loss, grad_logits,
                    param_grads, AdamState, adam_step, DrafterUpdater, OracleModel)
from oracle.update import ObjectiveWeights, kl_rl_schedule, loss_terms
from oracle.decode import LoggedTuple
from workloads import UpdateHyper, make_weights, workload, tiny_shape

N, V, D, R = 5, 16, 8, 2


def _batch(seed=0, tau=1.0):
    g = np.random.default_rng(seed)
    U = g.standard_normal((N, D))
    Ws = g.standard_normal((V, D)) * 0.5
    A = g.standard_normal((V, R)) * 0.3
    B = g.standard_normal((R, D)) * 0.3
    lg = g.standard_normal((N, V)) * 2
    a = g.integers(0, V, N)
    ys = g.integers(0, V, N)
    r = np.array([1, 1, 0, 1, 0], dtype=np.float64)
    return U, Ws, A, B, lg, a, ys, r


TERMS = {
    "kl": ObjectiveWeights(1, 0, 0, 0, 0, 0, 1.0),
    "kl_tau": ObjectiveWeights(1, 0, 0, 0, 0, 0, 2.5),
    "pg": ObjectiveWeights(0, 1, 0, 0, 0, 0, 1.0),
    "ce": ObjectiveWeights(0, 0, 1, 0, 0, 0, 1.0),
    "ent": ObjectiveWeights(0, 0, 0, 1, 0, 0, 1.0),
    "rl": ObjectiveWeights(0, 0, 0, 0, 1, 0, 1.0),
    "kl1": ObjectiveWeights(0, 0, 0, 0, 0, 1, 1.0),
    "mix": ObjectiveWeights(0.7, 0.4, 0.2, 0.05, 0.3, 0.11, 1.7),
}


@pytest.mark.parametrize("name", list(TERMS))
def test_grad_logits_finite_difference(name):
    U, Ws, A, B, lg, a, ys, r = _batch(1)
    w, b = TERMS[name], 0.37
    Z = head_logits(U, Ws, A, B, 0.8)
    G = grad_logits(Z, lg, a, ys, r, w, b)
    eps = 1e-6
    num = np.zeros_like(Z)
    for i in range(N):
        for j in range(V):
            Zp, Zm = Z.copy(), Z.copy()
            Zp[i, j] += eps
            Zm[i, j] -= eps
            num[i, j] = (total_loss(Zp, lg, a, ys, r, w, b)[0] -
                         total_loss(Zm, lg, a, ys, r, w, b)[0]) / (2 * eps)
    assert np.max(np.abs(num - G)) <= 1e-6 * max(1.0, np.max(np.abs(G)))
    assert np.abs(G).max() > 1e-4                      # the term is not vacuous
    np.testing.assert_allclose(G.sum(axis=1), 0.0, atol=1e-12)


@pytest.mark.parametrize("full", [False, True])
def test_param_grads_finite_difference(full):
    U, Ws, A, B, lg, a, ys, r = _batch(2)
    w, b, gamma = TERMS["mix"], 0.2, 0.8

    def L_of(Ws_, A_, B_):
        return total_loss(head_logits(U, Ws_, A_, B_, gamma), lg, a, ys, r, w, b)[0]

    G = grad_logits(head_logits(U, Ws, A, B, gamma), lg, a, ys, r, w, b)
    g = param_grads(G, U, A, B, gamma, full)
    eps = 1e-6
    targets = {"W_s": Ws} if full else {"A": A, "B": B}
    for name, P in targets.items():
        num = np.zeros_like(P)
        for idx in np.ndindex(P.shape):
            old = P[idx]
            P[idx] = old + eps
            lp = L_of(Ws, A, B)
            P[idx] = old - eps
            lm = L_of(Ws, A, B)
            P[idx] = old
            num[idx] = (lp - lm) / (2 * eps)
        rel = np.max(np.abs(num - g[name])) / np.max(np.abs(num))
        assert rel < 1e-6, (name, rel)


def test_closed_forms():
    Vn = 12
    Z = np.zeros((3, Vn))
    lg = np.zeros((3, Vn))
    t = loss_terms(Z, lg, np.array([0, 5, 11]), np.array([1, 2, 3]), 1.0)
    np.testing.assert_allclose(t["nll_a"], math.log(Vn))
    np.testing.assert_allclose(t["ent"], math.log(Vn))
    np.testing.assert_allclose(t["kl"], 0.0, atol=1e-15)
    # two classes: KL(Bern(p)||Bern(q)) by hand
    z = np.array([[math.log(0.3), math.log(0.7)]])
    l = np.array([[math.log(0.6), math.log(0.4)]])
    t = loss_terms(z, l, np.array([0]), np.array([0]), 1.0)
    ref = 0.3 * math.log(0.3 / 0.6) + 0.7 * math.log(0.7 / 0.4)
    assert abs(t["kl"][0] - ref) < 1e-14
    # temperature: q_tau = softmax(l / tau)
    t2 = loss_terms(z, 2 * l, np.array([0]), np.array([0]), 2.0)
    assert abs(t2["kl"][0] - ref) < 1e-14


def test_kl_gradient_vanishes_when_drafter_matches_teacher():
    g = np.random.default_rng(3)
    lg = g.standard_normal((4, 10))
    tau = 1.6
    Z = lg / tau + 3.0                                 # same distribution, shifted logits
    G = grad_logits(Z, lg, np.zeros(4, int), np.zeros(4, int), np.ones(4),
                    TERMS["kl_tau"].__class__(1, 0, 0, 0, 0, 0, tau), 0.0)
    assert np.abs(G).max() < 1e-15


def test_empty_accept_set_contributes_nothing():
    U, Ws, A, B, lg, a, ys, _ = _batch(4)
    r = np.zeros(N)
    Z = head_logits(U, Ws, A, B, 1.0)
    L, parts = total_loss(Z, lg, a, ys, r, TERMS["pg"], 0.0)
    G = grad_logits(Z, lg, a, ys, r, TERMS["pg"], 0.0)
    assert L == 0.0 and parts["pg"] == 0.0 and np.all(G == 0.0)


def test_schedule_breakpoints():
    h = UpdateHyper(objective="dvi", t_warmup=32, t_ramp=32, lambda0=1.0,
                    lambda_kl_min=0.1, lambda_pg_max=1.0)
    assert kl_rl_schedule(0, h) == (0.0, 1.0)
    assert kl_rl_schedule(31, h) == (0.0, 1.0)
    assert kl_rl_schedule(32, h) == (0.0, 1.0)                  # continuous at T_w
    pg, kl = kl_rl_schedule(48, h)                              # linear midpoint
    assert abs(pg - 0.5) < 1e-15 and abs(kl - 0.55) < 1e-15
    pg, kl = kl_rl_schedule(63, h)
    assert abs(pg - 31 / 32) < 1e-15 and abs(kl - (1 - 31 / 32 * 0.9)) < 1e-15
    assert kl_rl_schedule(64, h) == (1.0, 0.1)                  # continuous at T_w+T_ramp
    assert kl_rl_schedule(10 ** 6, h) == (1.0, 0.1)
    seq = [kl_rl_schedule(t, h) for t in range(100)]
    assert all(a[0] <= b[0] and a[1] >= b[1] for a, b in zip(seq, seq[1:]))
    w = objective_weights(10, h)
    assert w.w_rl == 0 and w.beta == 0                           # L_policy off in warmup
    w = objective_weights(32, h)
    assert abs(w.beta - h.beta0) < 1e-15
    assert objective_weights(10 ** 4, h).beta == pytest.approx(h.beta_min, abs=1e-12)
    assert objective_weights(80, h).w_rl == h.w_rl_max


def test_ablation_presets_are_single_term():
    for name, field in (("kl", "lam_kl"), ("pg", "w_rl"), ("ce", "lam_pg")):
        w = objective_weights(100, UpdateHyper(objective=name))
        on = [f.name for f in dataclasses.fields(w) if f.name != "tau" and getattr(w, f.name) != 0]
        assert on == [field]


def test_adam_first_steps_move_by_lr_sign():
    g = np.array([3.0, -0.25, 1e-3, -40.0])
    p = np.zeros(4)
    st = AdamState(np.zeros(4), np.zeros(4))
    adam_step(p, g, st, 0.01, 0.9, 0.999, 1e-12)
    np.testing.assert_allclose(p, -0.01 * np.sign(g), rtol=1e-8)
    adam_step(p, g, st, 0.01, 0.9, 0.999, 1e-12)
    np.testing.assert_allclose(p, -0.02 * np.sign(g), rtol=1e-8)


def test_adam_two_steps_hand_computed():
    """Two bias-corrected Adam steps with a changing gradient and an epsilon
    large enough to matter (lr 0.01, betas 0.9 / 0.999, eps 1e-3, p0 = 1):

    step 1, g = 2e-3:  m = 0.1 g = 2e-4, v = 0.001 g^2 = 4e-9,
      m^ = m / 0.1 = 2e-3, v^ = v / 0.001 = 4e-6, sqrt(v^) = 2e-3,
      p = 1 - 0.01 * 2e-3 / (2e-3 + 1e-3) = 1 - 0.02/3
    step 2, g = -1e-3: m = 0.9 * 2e-4 - 1e-4 = 8e-5,
      v = 0.999 * 4e-9 + 0.001 * 1e-6 = 4.996e-9,
      m^ = 8e-5 / 0.19 = 4.2105263157894737e-4,
      v^ = 4.996e-9 / 0.001999 = 2.4992496248124062e-6, sqrt(v^) = 1.5809015228066567e-3,
      p = p1 - 0.01 * m^ / (sqrt(v^) + 1e-3) = p1 - 1.6314168822724575e-3
    (worked by hand in decimal arithmetic).  Epsilon under the square root
    would give p1 = 0.99936880..., no bias correction p1 = 0.99811897..."""
    p = np.array([1.0])
    st = AdamState(np.zeros(1), np.zeros(1))
    adam_step(p, np.array([2e-3]), st, 0.01, 0.9, 0.999, 1e-3)
    assert p[0] == pytest.approx(0.99333333333333333, rel=1e-14)
    adam_step(p, np.array([-1e-3]), st, 0.01, 0.9, 0.999, 1e-3)
    assert p[0] == pytest.approx(0.99170191645106088, rel=1e-14)
    assert st.m[0] == pytest.approx(8e-5, rel=1e-12) and st.v[0] == pytest.approx(4.996e-9, rel=1e-12)


def _tuples(seed, n=6, d=32, V=64):
    g = np.random.default_rng(seed)
    return [LoggedTuple(seq=0, u=g.standard_normal(d), a=int(g.integers(V)),
                        logits=g.standard_normal(V), r=int(i < 4), i=i + 1, prev_id=0,
                        ystar=int(g.integers(V))) for i in range(n)]


def test_updater_sgd_step_and_baseline():
    shape = tiny_shape(d_model=32, vocab=64, n_layers=2, n_heads=2, n_kv_heads=2,
                       head_dim=16, d_ffn=48)
    w = workload("tiny").with_(shape=shape, lora_rank=3)
    m = OracleModel(make_weights(w, threads=2), shape, 0.5)
    m.lora_a = np.random.default_rng(1).standard_normal(m.lora_a.shape)
    A0, B0 = m.lora_a.copy(), m.lora_b.copy()
    h = UpdateHyper(objective="kl", optimizer="sgd", lr=0.1, baseline_rho=0.75)
    up = DrafterUpdater(m, h)
    tup = _tuples(0)
    info = up.update(tup)
    U = np.stack([t.u for t in tup])
    Lg = np.stack([t.logits for t in tup])
    a = np.array([t.a for t in tup]); ys = np.array([t.ystar for t in tup])
    r = np.array([t.r for t in tup], float)
    G = grad_logits(head_logits(U, m.w_s, A0, B0, 0.5), Lg, a, ys, r,
                    objective_weights(0, h), 0.0)
    g = param_grads(G, U, A0, B0, 0.5)
    np.testing.assert_allclose(m.lora_a, A0 - 0.1 * g["A"], rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(m.lora_b, B0 - 0.1 * g["B"], rtol=1e-12, atol=1e-15)
    assert up.b == pytest.approx(0.25 * 4 / 6) and up.t == 1
    up.update(tup)
    assert up.b == pytest.approx(0.75 * 0.25 * 4 / 6 + 0.25 * 4 / 6)


def test_planted_sign_error_is_caught(monkeypatch):
    """A flipped entropy-gradient sign must fail the finite-difference pin."""
    import oracle.update as upd
    U, Ws, A, B, lg, a, ys, r = _batch(5)
    w = TERMS["ent"]
    Z = head_logits(U, Ws, A, B, 1.0)
    good = grad_logits(Z, lg, a, ys, r, w, 0.0)
    orig = upd.grad_logits

    def bad(Z, lg, a, ys, r, w, b):
        return -orig(Z, lg, a, ys, r, w, b)

    monkeypatch.setattr(upd, "grad_logits", bad)
    eps = 1e-6
    Zp, Zm = Z.copy(), Z.copy()
    Zp[0, 0] += eps
    Zm[0, 0] -= eps
    num = (total_loss(Zp, lg, a, ys, r, w, 0.0)[0] - total_loss(Zm, lg, a, ys, r, w, 0.0)[0]) / (2 * eps)
    assert abs(num - good[0, 0]) < 1e-7
    assert abs(num - upd.grad_logits(Z, lg, a, ys, r, w, 0.0)[0, 0]) > 1e-4
