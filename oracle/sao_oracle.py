"""Plain, slow fp64 CPU oracle of the SAO per-token RL loss head.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
module. The CUDA product path (``paper_2607_07508_gb300``) never imports it and
shares no code, table or helper with it.

Every function writes out the definition it follows, in float64, with numpy
matmul as the only library step. Citations are to "Single-Rollout Asynchronous
Optimization for Agentic Reinforcement Learning" (arxiv 2607.07508):

* ``token_logprobs``      log pi_theta(a_t|s_t) of Eq. 1-2 (log-softmax of the
                          LM-head logits, gathered at the sampled token)
* ``token_logprobs_bwd``  gradient of sum_t G_t * log pi_theta(a_t|s_t) with
                          respect to the hidden states and the LM-head weight
* ``policy_loss``         Eq. 1-3: the ratio against the rollout policy (Eq. 2),
                          the strict double-sided mask f (Eq. 3) and the
                          token objective (Eq. 1); clip-ratio counts (§4.4)
* ``policy_loss_bwd``     d loss / d logp scaled by the incoming gradient
* ``advantages``          GAE of the Preliminaries, with the skip-observation
                          Bellman link of Eq. 4-5 and the length-adaptive
                          lambda of §4.1
* ``value_loss``          the value error (V - R)^2 of the Preliminaries (PPO),
                          with the explained-variance sums of §4.4
* ``step_advantages``     the step-level GAE variants of App. A.1 ("step
                          average" and "last-token prediction")
* ``clip_loss``           the clipped surrogate of the Preliminaries' unified
                          objective with asymmetric ("clip-higher") bounds, the
                          loss of the paper's GRPO / GRPO (w/ DIS) arms (§4.2)
* ``group_advantages``    GRPO's group-normalised advantage (Preliminaries)
* ``running_mean_advantages``  the running-mean reward baseline of the
                          single-rollout ablation (§4.3) and the online writing
                          comparison (§4.5)
* ``decoupled_loss``      the decoupled three-policy objective that DIS
                          simplifies (§3.1): a clipped ratio against the old
                          policy, weighted by the old/rollout ratio, with a
                          double-sided mask on that weight

Readings taken where the paper is silent or ambiguous (each one is listed with
its reason in the design notes):

R1  f(r) in Eq. 1 is a detached coefficient: the gradient is f(r)*A*grad(logp).
    The reported loss is the surrogate -(1/n) sum_t f(r_t)*A_t, which has that
    gradient and equals minus the masked mean advantage when old == new.
R2  The expectation over tokens is a token mean over the packed batch with
    denominator n_valid = number of action tokens (tokens with f = 0 still
    count), unless the caller passes its own normaliser n_norm > 0.
R3  Both bounds of Eq. 3 are strict; a ratio equal to a bound is masked. The
    in/out decision is taken on the fp32 log-ratio and the fp32 exponential
    (the precision the kernels use); values are fp64.
R4  A token whose log-ratio or advantage is not finite is masked and counted
    as non-finite; it still counts in n_valid.
R5  Advantages: the terminal reward sits on the last action token of the
    trajectory; the value after the last action token is 0; inside one action
    span ordinary GAE links adjacent tokens and across observation tokens the
    link jumps to the first token of the next action (Eq. 4-5), which is
    ordinary GAE over the action tokens only. Observation and prompt tokens get
    advantage 0 and return 0.
R6  Length-adaptive lambda: l is the trajectory's number of action tokens,
    lambda_b = 1 - 1/(alpha*l), clamped to [0, 1]; alpha <= 0 disables it.
R7  Returns are GAE with lambda_critic plus V; the value loss is the plain mean
    over action tokens of (V - ret)^2, no 1/2 factor and no clipping.
R13 Step-level GAE (App. A.1): a step is one conversation turn, i.e. a maximal
    run of action tokens inside a trajectory; the terminal reward is the
    reward of the last step; the step value after the last step is 0; every
    token of a step receives the step's advantage and the step's value target
    GAE(lambda_critic) + V(S); with "step average" every token of the step is
    a value-loss token, with "last-token" only the step's last token is.
R14 Clipped surrogate (Preliminaries): loss = -sum_t w_t min(r_t A_t,
    clip(r_t, 1-eps_low, 1+eps_high) A_t) with w_t = 1/(number of action
    tokens) ("token" normalisation) or 1/(|y_b| * number of trajectories with
    an action token) ("sequence": the per-sequence 1/|y| mean, then the batch
    mean). The ratio is taken against whatever log-probs the caller passes
    (pi_old for PPO/GRPO, pi_rollout for GRPO w/ DIS). A token is clipped when
    the min picks the clipped term strictly (A > 0 and r > 1+eps_high, or A < 0
    and r < 1-eps_low), decided in fp32; clipped tokens have zero gradient;
    non-finite tokens are masked as in R4.
R15 GRPO advantage: A_b = (R_b - mean_g) / sqrt(var_g + eps_stab) over the
    trajectories of b's group g (population variance), broadcast to b's action
    tokens; other tokens get 0.
R16 Running-mean baseline: trajectories are taken in batch order; the baseline
    of trajectory b is the mean of the (at most `window`) most recent rewards
    recorded for its prompt before b, 0 when there are none; A_b = R_b -
    baseline is broadcast to b's action tokens; then R_b enters the prompt's
    window. One shared prompt id gives the single global window of §4.5.
R17 Decoupled three-policy objective (§3.1 names its parts but writes no
    formula): r_t = pi_theta/pi_old corrects staleness and is clipped as in
    R14; w_t = pi_old/pi_rollout corrects the training/rollout mismatch and is
    kept only inside a strict band (w_low < w < w_high, the double-sided
    masking that §3.1 likens DIS to), else the token is masked. loss =
    -(1/n) sum_t w_t min(r_t A_t, clip(r_t, 1-eps_low, 1+eps_high) A_t) over
    kept action tokens, n as in R2; w is a detached coefficient, so
    d loss / d logp_t = -(1/n) w_t r_t A_t on unclipped kept tokens, else 0.
    All decisions in fp32, the mismatch test before the clip test.
"""
from __future__ import annotations

from typing import Dict, Tuple

import numpy as np

F64 = np.float64

FLAG_IN = 0
FLAG_LOW = 1
FLAG_HIGH = 2
FLAG_NONFINITE = 3
FLAG_MASKED = 4


def _f64(a) -> np.ndarray:
    """Exact upcast of a numpy array or torch tensor (fp32 or bf16) to fp64."""
    if hasattr(a, "detach"):
        a = a.detach().to("cpu")
        import torch
        a = a.to(torch.float64).numpy()
    return np.asarray(a, dtype=F64)


# ---------------------------------------------------------------------------
# Eq. 1-2: log pi_theta(a_t | s_t) from the LM head
# ---------------------------------------------------------------------------

def token_logprobs(H, W, y) -> Tuple[np.ndarray, np.ndarray]:
    """Log-probability of each sampled token under softmax(H W^T).

    z[t, v] = sum_k H[t, k] W[v, k]; lse[t] = log sum_v exp z[t, v];
    logp[t] = z[t, y[t]] - lse[t]. The log-sum-exp subtracts the row maximum
    before exponentiating (an exact identity) so large logits stay finite.
    Returns (logp, lse), both fp64 of length H.shape[0].
    """
    Hd, Wd = _f64(H), _f64(W)
    y = np.asarray(y, np.int64)
    n = Hd.shape[0]
    if n == 0:
        return np.zeros(0, F64), np.zeros(0, F64)
    Z = Hd @ Wd.T
    M = Z.max(axis=1)
    lse = M + np.log(np.exp(Z - M[:, None]).sum(axis=1))
    logp = Z[np.arange(n), y] - lse
    return logp, lse


def token_logprobs_bwd(H, W, y, lse, G) -> Tuple[np.ndarray, np.ndarray]:
    """Gradients of sum_t G[t] * logp[t] with respect to H and W.

    With p[t, v] = exp(z[t, v] - lse[t]), the derivative of logp[t] with
    respect to z[t, v] is 1[v == y[t]] - p[t, v]; so dZ[t, v] =
    G[t] * (1[v == y[t]] - p[t, v]), dH = dZ W and dW = dZ^T H.
    """
    Hd, Wd = _f64(H), _f64(W)
    y = np.asarray(y, np.int64)
    lse = _f64(lse)
    G = _f64(G)
    n = Hd.shape[0]
    Z = Hd @ Wd.T
    P = np.exp(Z - lse[:, None])
    dZ = -G[:, None] * P
    dZ[np.arange(n), y] += G
    dH = dZ @ Wd
    dW = dZ.T @ Hd
    return dH, dW


# ---------------------------------------------------------------------------
# Eq. 1-3: DIS ratio, strict double-sided mask, token objective
# ---------------------------------------------------------------------------

def mask_flags(logp, old_logp, adv, loss_mask, eps_low: float, eps_high: float) -> np.ndarray:
    """Per-token decision of Eq. 3, taken in fp32 (reading R3, R4).

    0: 1-eps_low < r < 1+eps_high (kept); 1: r <= 1-eps_low; 2: r >= 1+eps_high;
    3: log-ratio or advantage not finite; 4: not an action token.
    """
    lp32 = np.asarray(logp, np.float32)
    old32 = np.asarray(old_logp, np.float32)
    adv32 = np.asarray(adv, np.float32)
    m = np.asarray(loss_mask).astype(bool)
    with np.errstate(all="ignore"):
        d32 = (lp32 - old32).astype(np.float32)           # Eq. 2 exponent, fp32
        r32 = np.exp(d32).astype(np.float32)              # Eq. 2, fp32
        lo = np.float32(1.0) - np.float32(eps_low)
        hi = np.float32(1.0) + np.float32(eps_high)
        finite = np.isfinite(d32) & np.isfinite(adv32)
        flags = np.full(m.shape, FLAG_IN, np.uint8)
        flags[r32 >= hi] = FLAG_HIGH
        flags[r32 <= lo] = FLAG_LOW          # the lower test wins if both hold
    flags[~finite] = FLAG_NONFINITE
    flags[~m] = FLAG_MASKED
    return flags


def policy_loss(logp, old_logp, adv, loss_mask, eps_low: float, eps_high: float,
                n_norm: int = 0) -> Dict[str, object]:
    """Token-level DIS objective of Eq. 1 with the calibration f of Eq. 3.

    r_t = exp(logp_t - old_logp_t) (Eq. 2, rollout log-probs as the behaviour
    policy); f(r) = r if 1-eps_low < r < 1+eps_high else 0 (Eq. 3);
    loss = -(1/n) sum_t f(r_t) A_t; coef_t = d loss / d logp_t = -f(r_t) A_t / n
    with f detached (R1); n = n_norm if n_norm > 0 else the number of action
    tokens (R2). counts = [n_valid, n_low, n_high, n_nonfinite].
    """
    flags = mask_flags(logp, old_logp, adv, loss_mask, eps_low, eps_high)
    m = np.asarray(loss_mask).astype(bool)
    n_valid = int(m.sum())
    denom = int(n_norm) if n_norm > 0 else n_valid
    keep = flags == FLAG_IN
    with np.errstate(all="ignore"):
        r = np.exp(_f64(logp) - _f64(old_logp))
        f = np.where(keep, r, 0.0)
        contrib = np.where(keep, f * _f64(adv), 0.0)
    total = contrib.sum()
    loss = -total / denom if denom > 0 else 0.0
    coef = -contrib / denom if denom > 0 else np.zeros_like(contrib)
    counts = np.array([n_valid, int((flags == FLAG_LOW).sum()), int((flags == FLAG_HIGH).sum()),
                       int((flags == FLAG_NONFINITE).sum())], np.int64)
    return {"loss": float(loss), "coef": coef, "flags": flags, "counts": counts, "ratio": r}


def policy_loss_bwd(logp, old_logp, adv, loss_mask, eps_low, eps_high, n_norm, grad_loss) -> np.ndarray:
    """d(grad_loss * loss)/d logp_t = grad_loss * coef_t."""
    out = policy_loss(logp, old_logp, adv, loss_mask, eps_low, eps_high, n_norm)
    return out["coef"] * float(grad_loss)


def clip_ratio(counts) -> float:
    """Fraction of action tokens masked by f (the clip ratio monitored in §4.4)."""
    n = int(counts[0])
    return (int(counts[1]) + int(counts[2])) / n if n > 0 else 0.0


# ---------------------------------------------------------------------------
# GAE with the skip-observation link (Preliminaries; §3.2 Eq. 4-5; §4.1)
# ---------------------------------------------------------------------------

def trajectory_lambda(lam: float, alpha: float, n_actions: int) -> float:
    """lambda_policy = 1 - 1/(alpha * l) (length-adaptive, §4.1), reading R6."""
    if alpha <= 0.0:
        return float(lam)
    if n_actions <= 0:
        return 0.0
    return float(min(1.0, max(0.0, 1.0 - 1.0 / (alpha * n_actions))))


def _gae_backward(v: np.ndarray, rewards: np.ndarray, gamma: float, lam: float) -> np.ndarray:
    """Textbook backward GAE over one compacted action sequence.

    delta_j = r_j + gamma * V_{j+1} - V_j with V after the last step = 0;
    A_j = delta_j + gamma * lambda * A_{j+1}.
    """
    L = len(v)
    A = np.zeros(L, F64)
    nxt_A = 0.0
    for j in range(L - 1, -1, -1):
        v_next = v[j + 1] if j + 1 < L else 0.0
        delta = rewards[j] + gamma * v_next - v[j]
        nxt_A = delta + gamma * lam * nxt_A
        A[j] = nxt_A
    return A


def advantages(values, rewards, loss_mask, cu_seqlens, gamma: float, lam: float,
               lam_critic: float, alpha: float = 0.0) -> Tuple[np.ndarray, np.ndarray]:
    """Skip-observation token-level GAE and value targets for packed trajectories.

    For trajectory b with tokens [cu[b], cu[b+1]): keep its action tokens
    (loss_mask == 1) in order; their successor in the Bellman link is the next
    action token, skipping observation tokens (Eq. 4-5). The terminal reward
    R_b is the reward of the last action token (R5). Policy advantages use
    lambda_b (R6); returns are GAE(lambda_critic) + V (R7).
    Returns (adv, ret) as fp64 arrays over all N tokens.
    """
    v_all = _f64(values)
    R = _f64(rewards)
    m = np.asarray(loss_mask).astype(bool)
    cu = np.asarray(cu_seqlens, np.int64)
    N = len(v_all)
    adv = np.zeros(N, F64)
    ret = np.zeros(N, F64)
    for b in range(len(cu) - 1):
        idx = np.arange(cu[b], cu[b + 1])
        idx = idx[m[idx]]
        L = len(idx)
        if L == 0:
            continue
        v = v_all[idx]
        r = np.zeros(L, F64)
        r[-1] = R[b]
        lam_b = trajectory_lambda(lam, alpha, L)
        adv[idx] = _gae_backward(v, r, gamma, lam_b)
        ret[idx] = _gae_backward(v, r, gamma, lam_critic) + v
    return adv, ret


# ---------------------------------------------------------------------------
# value loss (Preliminaries, PPO) and explained variance (§4.4)
# ---------------------------------------------------------------------------

def value_loss(values, ret, loss_mask, n_norm: int = 0) -> Tuple[float, np.ndarray, np.ndarray]:
    """L_v = (1/n) sum_t m_t (V_t - ret_t)^2 over the action tokens
    (Preliminaries, the PPO value error), with n = n_norm if n_norm > 0, else
    the number of action tokens: the batch mean of the unsplit batch when
    data-parallel ranks share the batch's action-token count, as the policy
    loss's normaliser does.

    Returns (loss, dL/dV, ev_sums) with ev_sums = [sum m(R-V), sum m(R-V)^2,
    sum m R, sum m R^2] (R = ret) for the explained variance.
    """
    V = _f64(values)
    R = _f64(ret)
    m = np.asarray(loss_mask).astype(bool)
    n = int(n_norm) if n_norm > 0 else int(m.sum())
    d = np.where(m, V - R, 0.0)
    loss = float((d * d).sum() / n) if n > 0 else 0.0
    grad = 2.0 * d / n if n > 0 else np.zeros_like(d)
    e = np.where(m, R - V, 0.0)
    Rm = np.where(m, R, 0.0)
    ev = np.array([e.sum(), (e * e).sum(), Rm.sum(), (Rm * Rm).sum()], F64)
    return loss, grad, ev


def explained_variance(ev_sums, n: int) -> float:
    """EV = 1 - Var(R - V) / Var(R) over n action tokens (§4.4)."""
    if n <= 0:
        return float("nan")
    s1, s2, r1, r2 = (float(x) for x in ev_sums)
    var_e = s2 / n - (s1 / n) ** 2
    var_r = r2 / n - (r1 / n) ** 2
    return 1.0 - var_e / var_r if var_r > 0 else float("nan")


# ---------------------------------------------------------------------------
# step-level GAE variants (App. A.1)
# ---------------------------------------------------------------------------

STEP_AVERAGE = 0
STEP_LAST = 1


def step_spans(loss_mask, start: int, end: int):
    """Steps of the trajectory occupying tokens [start, end): maximal runs of
    action tokens, as (first, last + 1) pairs in order (reading R13)."""
    m = np.asarray(loss_mask).astype(bool)
    spans = []
    t = start
    while t < end:
        if m[t]:
            u = t
            while u < end and m[u]:
                u += 1
            spans.append((t, u))
            t = u
        else:
            t += 1
    return spans


def step_advantages(values, rewards, loss_mask, cu_seqlens, gamma: float, lam: float, lam_critic: float,
                    alpha: float = 0.0, mode: int = STEP_AVERAGE):
    """Step-wise GAE of App. A.1.

    V(S_i) = mean of the step's token values (STEP_AVERAGE) or the value of its
    last token (STEP_LAST); delta_i = r_i + gamma V(S_{i+1}) - V(S_i) with the
    terminal reward on the last step; A_i = sum_l (gamma lambda)^l delta_{i+l}
    with lambda = 1 - 1/(alpha * number of steps) when alpha > 0 (the
    length-adaptive rule counted in steps). Returns (adv, ret, value_mask)
    over all tokens: adv and ret broadcast to the step's tokens, value_mask =
    the tokens the value loss keeps (R13).
    """
    v_all = _f64(values)
    R = _f64(rewards)
    cu = np.asarray(cu_seqlens, np.int64)
    N = len(v_all)
    adv = np.zeros(N, F64)
    ret = np.zeros(N, F64)
    vmask = np.zeros(N, np.uint8)
    for b in range(len(cu) - 1):
        spans = step_spans(loss_mask, cu[b], cu[b + 1])
        n = len(spans)
        if n == 0:
            continue
        if mode == STEP_AVERAGE:
            vs = np.array([v_all[a:e].mean() for a, e in spans])
        else:
            vs = np.array([v_all[e - 1] for a, e in spans])
        r = np.zeros(n, F64)
        r[-1] = R[b]
        lam_b = trajectory_lambda(lam, alpha, n)
        A = _gae_backward(vs, r, gamma, lam_b)
        T = _gae_backward(vs, r, gamma, lam_critic) + vs
        for i, (a, e) in enumerate(spans):
            adv[a:e] = A[i]
            ret[a:e] = T[i]
            if mode == STEP_AVERAGE:
                vmask[a:e] = 1
            else:
                vmask[e - 1] = 1
    return adv, ret, vmask


# ---------------------------------------------------------------------------
# clipped surrogate of the PPO / GRPO arms (Preliminaries; §4.2 baselines)
# ---------------------------------------------------------------------------

NORM_TOKEN = 0
NORM_SEQUENCE = 1
CLIP_NONE = 0
CLIP_LOW = 1
CLIP_HIGH = 2


def clip_flags(logp, old_logp, adv, loss_mask, eps_low: float, eps_high: float) -> np.ndarray:
    """0: the unclipped term r*A is the min; 1: clipped at 1-eps_low (A < 0);
    2: clipped at 1+eps_high (A > 0); 3: non-finite; 4: not an action token.
    Decided in fp32 (R14)."""
    lp32 = np.asarray(logp, np.float32)
    old32 = np.asarray(old_logp, np.float32)
    adv32 = np.asarray(adv, np.float32)
    m = np.asarray(loss_mask).astype(bool)
    with np.errstate(all="ignore"):
        d32 = (lp32 - old32).astype(np.float32)
        r32 = np.exp(d32).astype(np.float32)
        lo = np.float32(1.0) - np.float32(eps_low)
        hi = np.float32(1.0) + np.float32(eps_high)
        flags = np.zeros(m.shape, np.uint8)
        flags[(adv32 > 0) & (r32 > hi)] = CLIP_HIGH
        flags[(adv32 < 0) & (r32 < lo)] = CLIP_LOW
        finite = np.isfinite(d32) & np.isfinite(adv32)
    flags[~finite] = FLAG_NONFINITE
    flags[~m] = FLAG_MASKED
    return flags


def clip_loss(logp, old_logp, adv, loss_mask, cu_seqlens, eps_low: float, eps_high: float,
              norm: int = NORM_TOKEN) -> Dict[str, object]:
    """Clipped surrogate with clip-higher bounds (R14).

    loss = -sum_t w_t min(r_t A_t, clip(r_t, 1-eps_low, 1+eps_high) A_t);
    coef_t = d loss / d logp_t = -w_t r_t A_t on unclipped tokens, else 0.
    counts = [n_action, n_clip_low, n_clip_high, n_nonfinite].
    """
    flags = clip_flags(logp, old_logp, adv, loss_mask, eps_low, eps_high)
    m = np.asarray(loss_mask).astype(bool)
    cu = np.asarray(cu_seqlens, np.int64)
    N = len(m)
    w = np.zeros(N, F64)
    if norm == NORM_TOKEN:
        n = int(m.sum())
        if n > 0:
            w[m] = 1.0 / n
    else:
        lens = [int(m[cu[b]:cu[b + 1]].sum()) for b in range(len(cu) - 1)]
        nseq = sum(1 for L in lens if L > 0)
        for b, L in enumerate(lens):
            if L > 0:
                sl = slice(cu[b], cu[b + 1])
                w[sl] = np.where(m[sl], 1.0 / (L * nseq), 0.0)
    with np.errstate(all="ignore"):
        r = np.exp(_f64(logp) - _f64(old_logp))
        A = _f64(adv)
        lo = float(np.float32(1.0) - np.float32(eps_low))
        hi = float(np.float32(1.0) + np.float32(eps_high))
        term = np.where(flags == CLIP_NONE, r * A,
                        np.where(flags == CLIP_LOW, lo * A, np.where(flags == CLIP_HIGH, hi * A, 0.0)))
        term = np.where(flags <= CLIP_HIGH, term, 0.0)
        coef = np.where(flags == CLIP_NONE, -w * r * A, 0.0)
    loss = -float((w * term).sum())
    counts = np.array([int(m.sum()), int((flags == CLIP_LOW).sum()), int((flags == CLIP_HIGH).sum()),
                       int((flags == FLAG_NONFINITE).sum())], np.int64)
    return {"loss": loss, "coef": coef, "flags": flags, "counts": counts}


def group_advantages(rewards, group_ids, loss_mask, cu_seqlens, eps_stab: float) -> np.ndarray:
    """GRPO advantage (R15): (R_b - mean_g) / sqrt(var_g + eps_stab)."""
    R = _f64(rewards)
    g = np.asarray(group_ids, np.int64)
    m = np.asarray(loss_mask).astype(bool)
    cu = np.asarray(cu_seqlens, np.int64)
    adv = np.zeros(len(m), F64)
    for b in range(len(R)):
        members = R[g == g[b]]
        mu = members.mean()
        var = ((members - mu) ** 2).mean()
        a = (R[b] - mu) / np.sqrt(var + eps_stab)
        sl = slice(cu[b], cu[b + 1])
        adv[sl] = np.where(m[sl], a, 0.0)
    return adv


# ---------------------------------------------------------------------------
# running-mean reward baseline (§4.3 ablation, §4.5 comparison)
# ---------------------------------------------------------------------------

def running_mean_advantages(rewards, prompt_ids, loss_mask, cu_seqlens, history, seen, window: int):
    """A_b = R_b - mean(recent rewards of b's prompt) (R16). `history`
    [P, window] and `seen` [P] are the per-prompt windows (ring buffers) and
    reward counts; copies are updated and returned with the advantages."""
    R = _f64(rewards)
    pid = np.asarray(prompt_ids, np.int64)
    m = np.asarray(loss_mask).astype(bool)
    cu = np.asarray(cu_seqlens, np.int64)
    hist = np.array(history, dtype=np.float64, copy=True)
    cnt = np.array(seen, dtype=np.int64, copy=True)
    adv = np.zeros(len(m), F64)
    for b in range(len(R)):
        p = pid[b]
        n = int(min(cnt[p], window))
        base = hist[p, :n].mean() if n > 0 else 0.0
        a = R[b] - base
        sl = slice(cu[b], cu[b + 1])
        adv[sl] = np.where(m[sl], a, 0.0)
        hist[p, cnt[p] % window] = R[b]
        cnt[p] += 1
    return adv, hist, cnt


# ---------------------------------------------------------------------------
# Decoupled three-policy objective (§3.1), reading R17
# ---------------------------------------------------------------------------

MIS_LOW = 5
MIS_HIGH = 6


def decoupled_flags(logp, prox_logp, rollout_logp, adv, loss_mask, eps_low: float, eps_high: float,
                    w_low: float, w_high: float) -> np.ndarray:
    """0 kept, unclipped; 1 / 2 clipped at 1-eps_low / 1+eps_high (as R14);
    3 non-finite; 4 not an action token; 5 w <= w_low; 6 w >= w_high.
    Decided in fp32 (R17)."""
    lp = np.asarray(logp, np.float32)
    px = np.asarray(prox_logp, np.float32)
    ro = np.asarray(rollout_logp, np.float32)
    a = np.asarray(adv, np.float32)
    m = np.asarray(loss_mask).astype(bool)
    with np.errstate(all="ignore"):
        d = (lp - px).astype(np.float32)        # log pi_theta/pi_old
        e = (px - ro).astype(np.float32)        # log pi_old/pi_rollout
        r = np.exp(d).astype(np.float32)
        w = np.exp(e).astype(np.float32)
        lo = np.float32(1.0) - np.float32(eps_low)
        hi = np.float32(1.0) + np.float32(eps_high)
        flags = np.zeros(m.shape, np.uint8)
        flags[(a > 0) & (r > hi)] = CLIP_HIGH
        flags[(a < 0) & (r < lo)] = CLIP_LOW
        flags[w >= np.float32(w_high)] = MIS_HIGH
        flags[w <= np.float32(w_low)] = MIS_LOW
        finite = np.isfinite(d) & np.isfinite(e) & np.isfinite(a)
    flags[~finite] = FLAG_NONFINITE
    flags[~m] = FLAG_MASKED
    return flags


def decoupled_loss(logp, prox_logp, rollout_logp, adv, loss_mask, eps_low: float, eps_high: float,
                   w_low: float, w_high: float, n_norm: int = 0) -> Dict[str, object]:
    """Decoupled PPO objective with the mismatch weight masked outside
    (w_low, w_high) (R17). counts = [n_action, n_clip_low, n_clip_high,
    n_nonfinite, n_mismatch_low, n_mismatch_high]."""
    flags = decoupled_flags(logp, prox_logp, rollout_logp, adv, loss_mask, eps_low, eps_high, w_low, w_high)
    m = np.asarray(loss_mask).astype(bool)
    n_action = int(m.sum())
    n = int(n_norm) if n_norm > 0 else n_action
    with np.errstate(all="ignore"):
        r = np.exp(_f64(logp) - _f64(prox_logp))
        w = np.exp(_f64(prox_logp) - _f64(rollout_logp))
        A = _f64(adv)
        lo = float(np.float32(1.0) - np.float32(eps_low))
        hi = float(np.float32(1.0) + np.float32(eps_high))
        term = np.where(flags == CLIP_NONE, r * A,
                        np.where(flags == CLIP_LOW, lo * A, np.where(flags == CLIP_HIGH, hi * A, 0.0)))
        contrib = np.where(flags <= CLIP_HIGH, w * term, 0.0)
        coef = np.where(flags == CLIP_NONE, -w * r * A / n, 0.0) if n > 0 else np.zeros(len(m))
    loss = -float(contrib.sum()) / n if n > 0 else 0.0
    counts = np.array([n_action, int((flags == CLIP_LOW).sum()), int((flags == CLIP_HIGH).sum()),
                       int((flags == FLAG_NONFINITE).sum()), int((flags == MIS_LOW).sum()),
                       int((flags == MIS_HIGH).sum())], np.int64)
    return {"loss": loss, "coef": coef, "flags": flags, "counts": counts}
