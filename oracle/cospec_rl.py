"""Reward shaping and advantages of CoSpec's RL stage (Sec. 3.4) -- TEST
INFRASTRUCTURE ONLY: a plain float64 restatement, one equation at a time, used
by the tests to check the CUDA path.  Shares no code with it.

A batch holds prompt groups; group x owns rollouts group_off[x] .. group_off[x+1]-1,
rollout m owns rounds round_off[m] .. round_off[m+1]-1, and round r carries, for
draft positions i = 1..K (array index i-1): the match flags Delta_i (Eq. 3),
the actions a_i (1 = keep the draft token; 1 at matches) and
ell_i = log p_T(y_hat_i | ...) (Eq. 23).

Readings where the paper is silent: sigma_x is the population standard
deviation over the group; epsilon is a call parameter (1e-6 by default); a
round without a mismatch contributes nothing (as the paper says); when a failed
rollout's penalties sum to 0 its decisions get advantage 0; the entropy and KL
terms of the objective are the Bernoulli ones of pi_theta(a = 1) at every
effective decision, summed like the clipped surrogate.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np


@dataclass
class RLParams:
    alpha: float = 1.0        # risk penalty weight (App. C: 1.0)
    beta: float = 0.25        # rejection penalty (App. C: 0.25)
    eta_fail: float = 0.5     # all-incorrect group weight (App. C: 0.5)
    eps: float = 1e-6
    clip_eps: float = 0.2     # PPO clip range (App. C: 0.2)
    beta_h: float = 0.01      # entropy coefficient (App. C: 0.01)
    beta_kl: float = 0.02     # KL coefficient (App. C: 0.02)


def round_quantities(match, accept, K: int):
    """For one round: (s, i_star, i_rej, rho, effective set I_r), 1-based
    positions.  s = first i with Delta_i = 0 and a_i = 0, else K+1 (Eq. 15);
    i_star = first mismatch (None when there is none); i_rej = s when a
    mismatch is rejected, else the sentinel K+1; rho = (s - i*) / ((K+1) - i*);
    I_r = {i : Delta_i = 0, i <= min(s, K)}."""
    s = K + 1
    for i in range(1, K + 1):
        if match[i - 1] == 0 and accept[i - 1] == 0:
            s = i
            break
    mism = [i for i in range(1, K + 1) if match[i - 1] == 0]
    if not mism:
        return s, None, K + 1, None, []
    i_star = mism[0]
    i_rej = s if s <= K else K + 1
    rho = (s - i_star) / ((K + 1) - i_star)
    eff = [i for i in mism if i <= min(s, K)]
    return s, i_star, i_rej, rho, eff


def decision_rewards(correct: bool, match, accept, ell, K: int, prm: RLParams):
    """g_{r,i} for the effective decisions of one round: rho_r for a correct
    rollout; -alpha |ell_i| for accepted mismatches before the first rejection
    and -beta for the rejection itself for an incorrect one (Eq. failure
    penalty).  Returns ({i: g}, rho)."""
    s, i_star, i_rej, rho, eff = round_quantities(match, accept, K)
    g = {}
    for i in eff:
        if correct:
            g[i] = rho
        else:
            acc = accept[i - 1] == 1 and i < i_rej
            rej = i == i_rej and i_rej <= K
            g[i] = -prm.alpha * abs(float(ell[i - 1])) * acc - prm.beta * rej
    return g, rho


def bernoulli_entropy(p: float) -> float:
    h = 0.0
    for q in (p, 1.0 - p):
        if q > 0.0:
            h -= q * math.log(q)
    return h


def bernoulli_kl(p: float, q: float) -> float:
    k = 0.0
    for a, b in ((p, q), (1.0 - p, 1.0 - q)):
        if a > 0.0:
            k += a * math.log(a / b)
    return k


def rl_advantages(group_off, correct, round_off, K, match, accept, ell, prm: RLParams,
                  ratio=None, p_new=None, p_ref=None):
    """All outputs of the RL stage for a batch (Sec. 3.4):
    g [R][K] (0 outside effective decisions), eff [R][K], rho [R] (NaN without a
    mismatch), J [M], Jbar [M], adv [M], adv_dec [R][K], and, when ratio /
    p_new / p_ref [R][K] are given, (surrogate, entropy, kl, loss) with
    loss = -surrogate - beta_H entropy + beta_KL kl."""
    group_off = np.asarray(group_off); round_off = np.asarray(round_off)
    match = np.asarray(match); accept = np.asarray(accept); ell = np.asarray(ell, dtype=np.float64)
    M = len(correct)
    Rt = int(round_off[-1]) if M else 0
    g = np.zeros((Rt, K)); eff = np.zeros((Rt, K), dtype=np.uint8)
    rho = np.full(Rt, np.nan)
    J = np.zeros(M); sabs = np.zeros(M)
    for m in range(M):
        for r in range(int(round_off[m]), int(round_off[m + 1])):
            gr, rr = decision_rewards(bool(correct[m]), match[r], accept[r], ell[r], K, prm)
            if rr is not None:
                rho[r] = rr
            for i, v in gr.items():
                g[r, i - 1] = v
                eff[r, i - 1] = 1
                J[m] += v                               # J = sum_r sum_{i in I_r} g_{r,i}
                sabs[m] += abs(v)
    Jbar = J.copy(); adv = np.zeros(M)
    for x in range(len(group_off) - 1):
        ms = list(range(int(group_off[x]), int(group_off[x + 1])))
        if not ms:
            continue
        pos = [m for m in ms if correct[m]]
        neg = [m for m in ms if not correct[m]]
        eta = 1.0
        if pos and neg:
            gamma = sum(abs(J[m]) for m in neg) / (sum(J[m] for m in pos) + prm.eps)   # Eq. gamma
            for m in pos:
                Jbar[m] = gamma * J[m]
        elif not pos:
            eta = prm.eta_fail
        vals = np.array([Jbar[m] for m in ms])
        mu = vals.mean()
        sigma = math.sqrt(((vals - mu) ** 2).mean())
        for m in ms:
            adv[m] = eta * (Jbar[m] - mu) / (sigma + prm.eps)                             # Eq. adv
    adv_dec = np.zeros((Rt, K))
    for m in range(M):
        for r in range(int(round_off[m]), int(round_off[m + 1])):
            for i in range(K):
                if not eff[r, i]:
                    continue
                if correct[m]:
                    adv_dec[r, i] = rho[r] * adv[m]
                else:
                    adv_dec[r, i] = (abs(g[r, i]) / sabs[m] * adv[m]) if sabs[m] > 0 else 0.0
    out = dict(g=g, eff=eff, rho=rho, J=J, Jbar=Jbar, adv=adv, adv_dec=adv_dec)
    if ratio is not None:
        ratio = np.asarray(ratio, dtype=np.float64)
        p_new = np.asarray(p_new, dtype=np.float64); p_ref = np.asarray(p_ref, dtype=np.float64)
        surr = ent = kl = 0.0
        for r in range(Rt):
            for i in range(K):
                if not eff[r, i]:
                    continue
                a = adv_dec[r, i]
                rc = min(max(ratio[r, i], 1.0 - prm.clip_eps), 1.0 + prm.clip_eps)
                surr += min(ratio[r, i] * a, rc * a)
                ent += bernoulli_entropy(p_new[r, i])
                kl += bernoulli_kl(p_new[r, i], p_ref[r, i])
        out["loss_terms"] = (surr, ent, kl, -surr - prm.beta_h * ent + prm.beta_kl * kl)
    return out
