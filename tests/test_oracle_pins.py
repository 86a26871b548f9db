"""Pins of the fp64 oracle against facts the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a brute-force
loop written from the definition, a closed form, an invariant, a special case
that reduces to a library routine, or a finite-difference derivative. Each is
chosen so that a plausible slip (dropped term, wrong sign or index, transposed
operand, non-strict bound, wrong successor across an observation span) fails.
"""
import json
import math
import os

import numpy as np
import pytest

from oracle import sao_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_hyperparams.json")


def _rng(seed):
    return np.random.Generator(np.random.PCG64(seed))


# ---------------------------------------------------------------------------
# log-probs (Eq. 1-2)
# ---------------------------------------------------------------------------

def test_logprobs_bruteforce_loops():
    """Explicit loops over t, v, k with math.fsum; non-square shapes catch a
    transposed operand or a wrong gather index."""
    r = _rng(1)
    N, h, V = 5, 3, 7
    H = r.normal(size=(N, h))
    W = r.normal(size=(V, h))
    y = r.integers(0, V, size=N)
    logp, lse = O.token_logprobs(H, W, y)
    for t in range(N):
        z = [math.fsum(H[t, k] * W[v, k] for k in range(h)) for v in range(V)]
        s = math.fsum(math.exp(zv) for zv in z)
        assert abs(lse[t] - math.log(s)) < 1e-12
        assert abs(logp[t] - (z[y[t]] - math.log(s))) < 1e-12


def test_logprobs_normalise_to_one():
    """sum_v exp(log pi(v|s_t)) = 1 for every row."""
    r = _rng(2)
    N, h, V = 6, 8, 33
    H = r.normal(size=(N, h)) * 2.0
    W = r.normal(size=(V, h))
    tot = np.zeros(N)
    for v in range(V):
        lp, _ = O.token_logprobs(H, W, np.full(N, v))
        tot += np.exp(lp)
    assert np.allclose(tot, 1.0, atol=1e-13, rtol=0)


def test_logprobs_zero_weight_uniform():
    N, h, V = 4, 5, 151936
    H = _rng(3).normal(size=(N, h))
    W = np.zeros((V, h))
    lp, _ = O.token_logprobs(H, W, np.arange(N))
    assert np.allclose(lp, -math.log(V), rtol=1e-15, atol=0)


def test_logprobs_single_vocab_is_zero():
    H = _rng(4).normal(size=(3, 4))
    W = _rng(5).normal(size=(1, 4))
    lp, _ = O.token_logprobs(H, W, np.zeros(3, np.int64))
    assert np.all(np.abs(lp) < 1e-15)


def test_logprobs_large_logits_match_library():
    """Logits of size ~1e3 stay finite and match scipy's log_softmax."""
    from scipy.special import log_softmax
    r = _rng(6)
    N, h, V = 7, 4, 50
    H = r.normal(size=(N, h)) * 300.0
    W = r.normal(size=(V, h))
    y = r.integers(0, V, size=N)
    lp, _ = O.token_logprobs(H, W, y)
    ref = log_softmax(H @ W.T, axis=1)[np.arange(N), y]
    assert np.all(np.isfinite(lp)) and np.all(lp <= 0)
    assert np.allclose(lp, ref, rtol=1e-12, atol=1e-9)


# ---------------------------------------------------------------------------
# log-prob gradients
# ---------------------------------------------------------------------------

def _logp_objective(H, W, y, G):
    lp, _ = O.token_logprobs(H, W, y)
    return float(np.dot(G, lp))


def test_logprobs_bwd_finite_differences():
    r = _rng(7)
    N, h, V = 4, 3, 5
    H = r.normal(size=(N, h))
    W = r.normal(size=(V, h))
    y = r.integers(0, V, size=N)
    G = r.normal(size=N)
    G[1] = 0.0
    _, lse = O.token_logprobs(H, W, y)
    dH, dW = O.token_logprobs_bwd(H, W, y, lse, G)
    eps = 1e-6
    for X, dX in ((H, dH), (W, dW)):
        num = np.zeros_like(X)
        for idx in np.ndindex(X.shape):
            old = X[idx]
            X[idx] = old + eps
            fp = _logp_objective(H, W, y, G)
            X[idx] = old - eps
            fm = _logp_objective(H, W, y, G)
            X[idx] = old
            num[idx] = (fp - fm) / (2 * eps)
        assert np.allclose(num, dX, atol=1e-8, rtol=1e-6)


def test_logprobs_bwd_invariants():
    r = _rng(8)
    N, h, V = 9, 6, 20
    H = r.normal(size=(N, h))
    W = r.normal(size=(V, h))
    y = r.integers(0, V, size=N)
    G = r.normal(size=N)
    G[3] = 0.0
    _, lse = O.token_logprobs(H, W, y)
    dH, dW = O.token_logprobs_bwd(H, W, y, lse, G)
    # every row of dZ sums to zero, so the vocab rows of dW sum to zero
    assert np.allclose(dW.sum(axis=0), 0.0, atol=1e-12)
    # a row with G = 0 contributes nothing
    assert np.all(dH[3] == 0.0)
    # identical weight rows: dH = w * sum_v dZ = 0
    W2 = np.tile(r.normal(size=(1, h)), (V, 1))
    _, lse2 = O.token_logprobs(H, W2, y)
    dH2, _ = O.token_logprobs_bwd(H, W2, y, lse2, G)
    assert np.allclose(dH2, 0.0, atol=1e-12)


def test_logprobs_bwd_torch_autograd():
    torch = pytest.importorskip("torch")
    r = _rng(9)
    N, h, V = 6, 5, 11
    H = r.normal(size=(N, h))
    W = r.normal(size=(V, h))
    y = r.integers(0, V, size=N)
    G = r.normal(size=N)
    _, lse = O.token_logprobs(H, W, y)
    dH, dW = O.token_logprobs_bwd(H, W, y, lse, G)
    Ht = torch.tensor(H, requires_grad=True)
    Wt = torch.tensor(W, requires_grad=True)
    lp = torch.log_softmax(Ht @ Wt.T, dim=1)[torch.arange(N), torch.tensor(y)]
    (lp * torch.tensor(G)).sum().backward()
    assert np.allclose(Ht.grad.numpy(), dH, atol=1e-12)
    assert np.allclose(Wt.grad.numpy(), dW, atol=1e-12)


# ---------------------------------------------------------------------------
# policy loss (Eq. 1-3)
# ---------------------------------------------------------------------------

def _loss_inputs(seed, N=64):
    r = _rng(seed)
    logp = (-r.exponential(2.0, size=N)).astype(np.float32)
    old = (logp + r.normal(0, 0.1, size=N)).astype(np.float32)
    adv = r.normal(size=N).astype(np.float32)
    m = (r.random(N) < 0.8).astype(np.uint8)
    return logp, old, adv, m


def test_policy_loss_old_equals_new():
    """old == new: every action token is in bound (r = 1) and the loss is minus
    the masked mean advantage."""
    logp, _, adv, m = _loss_inputs(10)
    out = O.policy_loss(logp, logp, adv, m, 0.2, 0.28)
    n = m.sum()
    assert np.all(out["flags"][m == 1] == O.FLAG_IN)
    assert np.all(out["flags"][m == 0] == O.FLAG_MASKED)
    assert abs(out["loss"] - (-(adv.astype(np.float64) * m).sum() / n)) < 1e-12
    assert np.allclose(out["coef"], -(adv.astype(np.float64) * m) / n, atol=1e-15)
    assert list(out["counts"]) == [n, 0, 0, 0]


def test_policy_loss_hand_example():
    """Four action tokens with eps = (0.2, 0.28): ratios e^0, e^0.3, e^-0.3, e^0.2.
    e^0.3 = 1.35 >= 1.28 is masked high, e^-0.3 = 0.741 <= 0.8 is masked low."""
    logp = np.array([-1.0, -0.7, -1.3, -0.8], np.float32)
    old = np.array([-1.0, -1.0, -1.0, -1.0], np.float32)
    adv = np.array([0.5, 2.0, -1.0, -0.25], np.float32)
    m = np.ones(4, np.uint8)
    out = O.policy_loss(logp, old, adv, m, 0.2, 0.28)
    assert list(out["flags"]) == [0, 2, 1, 0]
    r3 = math.exp(float(np.float32(-0.8)) - float(np.float32(-1.0)))
    want = -(1.0 * 0.5 + r3 * -0.25) / 4.0
    assert abs(out["loss"] - want) < 1e-12
    assert list(out["counts"]) == [4, 1, 1, 0]


def test_policy_loss_bounds_are_strict():
    """A ratio exactly equal to 1-eps_low or 1+eps_high is masked (Eq. 3 uses
    strict inequalities); the next representable ratio inward is kept."""
    for d in (np.float32(-0.25), np.float32(-0.6)):
        r = np.float32(np.exp(np.float32(d)))
        eps_l = float(np.float32(1.0) - r)                # exact (Sterbenz)
        assert np.float32(1.0) - np.float32(eps_l) == r
        f = O.mask_flags([d], [0.0], [1.0], [1], eps_l, 0.5)
        assert f[0] == O.FLAG_LOW
        d_in = np.nextafter(d, np.float32(0.0))
        f2 = O.mask_flags([d_in], [0.0], [1.0], [1], eps_l, 0.5)
        if np.float32(np.exp(d_in)) > r:
            assert f2[0] == O.FLAG_IN
    for d in (np.float32(0.25), np.float32(0.6)):
        r = np.float32(np.exp(np.float32(d)))
        eps_h = float(r - np.float32(1.0))
        assert np.float32(1.0) + np.float32(eps_h) == r
        f = O.mask_flags([d], [0.0], [1.0], [1], 0.5, eps_h)
        assert f[0] == O.FLAG_HIGH
        d_in = np.nextafter(d, np.float32(0.0))
        f2 = O.mask_flags([d_in], [0.0], [1.0], [1], 0.5, eps_h)
        if np.float32(np.exp(d_in)) < r:
            assert f2[0] == O.FLAG_IN


def test_policy_loss_no_bounds_is_ratio_weighted_mean():
    logp, old, adv, m = _loss_inputs(11)
    out = O.policy_loss(logp, old, adv, m, 1e30, 1e30)
    r = np.exp(logp.astype(np.float64) - old.astype(np.float64))
    want = -(r * adv * m).sum() / m.sum()
    assert abs(out["loss"] - want) < 1e-12 * max(1.0, abs(want))


def test_policy_loss_finite_difference_matches_coef():
    logp, old, adv, m = _loss_inputs(12, N=24)
    eps_l, eps_h = 0.3, 5.0
    out = O.policy_loss(logp, old, adv, m, eps_l, eps_h)
    lp = logp.astype(np.float64)
    step = 1e-7
    for t in range(len(lp)):
        r = math.exp(lp[t] - float(old[t]))
        if abs(r - (1 - eps_l)) < 1e-4 or abs(r - (1 + eps_h)) < 1e-4:
            continue
        a = lp.copy()
        a[t] += step
        b = lp.copy()
        b[t] -= step
        fa = O.policy_loss(a, old, adv, m, eps_l, eps_h)["loss"]
        fb = O.policy_loss(b, old, adv, m, eps_l, eps_h)["loss"]
        assert abs((fa - fb) / (2 * step) - out["coef"][t]) < 1e-7


def test_policy_loss_nonfinite_and_mask():
    logp = np.array([-1.0, -1.0, -1.0, -1.0, -1.0], np.float32)
    old = np.array([-np.inf, -1.0, np.nan, -1.0, -1.0], np.float32)
    adv = np.array([1.0, np.nan, 1.0, 1.0, 1.0], np.float32)
    m = np.array([1, 1, 1, 0, 1], np.uint8)
    out = O.policy_loss(logp, old, adv, m, 0.2, 0.28)
    assert list(out["flags"]) == [3, 3, 3, 4, 0]
    assert list(out["counts"]) == [4, 0, 0, 3]
    assert abs(out["loss"] - (-1.0 / 4)) < 1e-15


def test_policy_loss_external_normaliser_and_grad_scale():
    logp, old, adv, m = _loss_inputs(13)
    a = O.policy_loss(logp, old, adv, m, 0.2, 0.28)
    b = O.policy_loss(logp, old, adv, m, 0.2, 0.28, n_norm=1000)
    assert abs(b["loss"] * 1000 - a["loss"] * m.sum()) < 1e-12
    g = O.policy_loss_bwd(logp, old, adv, m, 0.2, 0.28, 0, 2.5)
    assert np.allclose(g, 2.5 * a["coef"], atol=0, rtol=0)


def test_policy_loss_eps_low_one_disables_lower_mask():
    logp = np.array([-30.0, -5.0], np.float32)
    old = np.zeros(2, np.float32)
    out = O.policy_loss(logp, old, np.ones(2, np.float32), np.ones(2, np.uint8), 1.0, 0.5)
    assert list(out["flags"]) == [0, 0]


def test_clip_ratio_hand_counts_and_empty_batch():
    """§4.4's clip ratio: the share of action tokens that f masks by a bound.
    The hand example above masks one token low and one high out of four;
    non-finite tokens are masked but not clipped; no action token gives 0."""
    logp = np.array([-1.0, -0.7, -1.3, -0.8], np.float32)
    old = np.full(4, -1.0, np.float32)
    out = O.policy_loss(logp, old, np.array([0.5, 2.0, -1.0, -0.25], np.float32), np.ones(4, np.uint8), 0.2, 0.28)
    assert O.clip_ratio(out["counts"]) == 0.5
    assert O.clip_ratio([4, 0, 0, 3]) == 0.0
    assert O.clip_ratio([7, 2, 0, 5]) == 2 / 7
    assert O.clip_ratio([0, 0, 0, 0]) == 0.0
    assert O.clip_ratio(np.zeros(4, np.int64)) == 0.0


def test_clip_ratio_brute_force():
    """Counted token by token in fp64 on ratios kept 1e-3 away from both
    bounds: clipped action tokens over all action tokens."""
    r = _rng(31)
    N = 400
    ratio = np.exp(r.normal(0.0, 0.5, size=N))
    el, eh = 0.3, 0.4
    keep = (np.abs(ratio - (1 - el)) > 1e-3) & (np.abs(ratio - (1 + eh)) > 1e-3)
    ratio = ratio[keep]
    old = np.zeros(len(ratio), np.float32)
    logp = np.log(ratio).astype(np.float32)
    m = (r.random(len(ratio)) < 0.8).astype(np.uint8)
    out = O.policy_loss(logp, old, np.ones(len(ratio), np.float32), m, el, eh)
    clipped = sum(1 for t in range(len(ratio)) if m[t] and (ratio[t] <= 1 - el or ratio[t] >= 1 + eh))
    assert 0 < clipped < m.sum()
    assert O.clip_ratio(out["counts"]) == clipped / int(m.sum())


def test_policy_loss_paper_bounds():
    hp = json.load(open(GOLDEN))
    for key in ("clip_reasoning", "clip_coding"):
        el, eh = hp[key]["eps_low"], hp[key]["eps_high"]
        d = np.array([math.log(1 - el) - 0.01, math.log(1 - el) + 0.01,
                      math.log(1 + eh) - 0.01, math.log(1 + eh) + 0.01], np.float32)
        f = O.mask_flags(d, np.zeros(4), np.ones(4), np.ones(4), el, eh)
        assert list(f) == [1, 0, 0, 2]


# ---------------------------------------------------------------------------
# skip-observation GAE (Preliminaries, Eq. 4-5, §4.1)
# ---------------------------------------------------------------------------

def _traj(seed, L, obs_frac=0.3):
    r = _rng(seed)
    m = (r.random(L) >= obs_frac).astype(np.uint8)
    v = r.normal(0.4, 0.2, size=L)
    return m, v


def _explicit_sum_gae(v_act, R, gamma, lam):
    """A_t = sum_l (gamma lambda)^l delta_{t+l} over the action sequence, written
    as the explicit sum of the Preliminaries (not as a recursion)."""
    L = len(v_act)
    vn = np.append(v_act[1:], 0.0)
    rew = np.zeros(L)
    rew[-1] = R
    delta = rew + gamma * vn - v_act
    return np.array([sum((gamma * lam) ** l * delta[t + l] for l in range(L - t)) for t in range(L)])


def test_gae_gamma_lambda_one_telescopes():
    """gamma = lambda = 1: A_t = R - V_t on every action token (with or without
    observation spans in between); observation tokens get 0."""
    lens = [37, 1, 0, 64]
    ms, vs = [], []
    for i, L in enumerate(lens):
        m, v = _traj(20 + i, L)
        ms.append(m)
        vs.append(v)
    m = np.concatenate(ms)
    v = np.concatenate(vs)
    cu = np.concatenate([[0], np.cumsum(lens)])
    R = np.array([1.0, 0.0, 1.0, 1.0])
    adv, ret = O.advantages(v, R, m, cu, 1.0, 1.0, 1.0)
    for b in range(len(lens)):
        sl = slice(cu[b], cu[b + 1])
        mb = m[sl].astype(bool)
        assert np.allclose(adv[sl][mb], R[b] - v[sl][mb], atol=1e-13)
        assert np.all(adv[sl][~mb] == 0) and np.all(ret[sl][~mb] == 0)
        assert np.allclose(ret[sl][mb], R[b], atol=1e-13)


def test_gae_lambda_zero_is_td_residual_across_observations():
    """gamma*lambda = 0: A equals delta, whose successor value skips observation
    tokens (Eq. 5)."""
    m = np.array([1, 1, 0, 0, 1, 0, 1, 1, 0], np.uint8)
    v = np.array([0.1, 0.2, 9.0, 9.0, 0.3, 9.0, 0.4, 0.5, 9.0])
    gamma = 0.9
    adv, _ = O.advantages(v, np.array([1.0]), m, np.array([0, 9]), gamma, 0.0, 1.0)
    act = np.flatnonzero(m)
    want = {0: gamma * 0.2 - 0.1, 1: gamma * 0.3 - 0.2, 4: gamma * 0.4 - 0.3,
            6: gamma * 0.5 - 0.4, 7: 1.0 + 0.0 - 0.5}
    for t in act:
        assert abs(adv[t] - want[t]) < 1e-15
    assert np.all(adv[m == 0] == 0)


def test_gae_matches_explicit_sum_without_observations():
    m = np.ones(40, np.uint8)
    v = _rng(30).normal(0.4, 0.2, size=40)
    for gamma, lam in ((1.0, 0.95), (0.97, 0.9), (0.5, 1.0)):
        adv, _ = O.advantages(v, np.array([1.0]), m, np.array([0, 40]), gamma, lam, 1.0)
        assert np.allclose(adv, _explicit_sum_gae(v, 1.0, gamma, lam), atol=1e-13)


def test_gae_inserting_observations_leaves_actions_unchanged():
    """Eq. 4-5: the Bellman link jumps over observation tokens, so adding
    observation tokens (with arbitrary values) changes no action-token output."""
    r = _rng(31)
    L = 50
    v = r.normal(0.4, 0.2, size=L)
    a0, ret0 = O.advantages(v, np.array([1.0]), np.ones(L, np.uint8), np.array([0, L]), 0.99, 0.9, 1.0)
    ins = np.sort(r.choice(np.arange(1, L), size=8, replace=False))
    v2, m2 = [], []
    for t in range(L):
        if t in ins:
            for _ in range(3):
                v2.append(r.normal(5, 3))
                m2.append(0)
        v2.append(v[t])
        m2.append(1)
    v2.append(-7.0)                # trailing observation after the last action
    m2.append(0)
    v2, m2 = np.array(v2), np.array(m2, np.uint8)
    a1, ret1 = O.advantages(v2, np.array([1.0]), m2, np.array([0, len(v2)]), 0.99, 0.9, 1.0)
    assert np.allclose(a1[m2 == 1], a0, atol=1e-13)
    assert np.allclose(ret1[m2 == 1], ret0, atol=1e-13)


def test_gae_critic_lambda_one_is_discounted_reward_to_go():
    m, v = _traj(32, 30)
    L = int(m.sum())
    gamma = 0.9
    _, ret = O.advantages(v, np.array([1.0]), m, np.array([0, 30]), gamma, 0.5, 1.0)
    k = np.arange(L)[::-1]
    assert np.allclose(ret[m == 1], gamma ** k, atol=1e-13)


def test_gae_length_adaptive_lambda():
    """gamma = 1, V = 0, R = 1: A_j = lambda_b^(L-1-j) with lambda_b = 1 - 1/(1.5 L)."""
    hp = json.load(open(GOLDEN))
    alpha = hp["length_adaptive_gae"]["alpha"]
    for L in (1, 2, 7, 100):
        v = np.zeros(L)
        adv, _ = O.advantages(v, np.array([1.0]), np.ones(L, np.uint8), np.array([0, L]),
                              1.0, 0.123, 1.0, alpha)
        lb = max(0.0, 1.0 - 1.0 / (alpha * L))
        assert np.allclose(adv, lb ** np.arange(L)[::-1], atol=1e-14)


def test_gae_trajectories_are_independent():
    lens = [10, 0, 7, 12]
    ms, vs = zip(*[_traj(40 + i, L) for i, L in enumerate(lens)])
    m, v = np.concatenate(ms), np.concatenate(vs)
    cu = np.concatenate([[0], np.cumsum(lens)])
    R = np.array([1.0, 1.0, 0.0, 1.0])
    adv, ret = O.advantages(v, R, m, cu, 0.95, 0.9, 1.0)
    for b in range(len(lens)):
        sl = slice(cu[b], cu[b + 1])
        a1, r1 = O.advantages(v[sl], R[b:b + 1], m[sl], np.array([0, lens[b]]), 0.95, 0.9, 1.0)
        assert np.allclose(adv[sl], a1, atol=0) and np.allclose(ret[sl], r1, atol=0)


def test_gae_no_action_tokens():
    m = np.zeros(5, np.uint8)
    adv, ret = O.advantages(np.ones(5), np.array([1.0]), m, np.array([0, 5]), 1.0, 1.0, 1.0, 1.5)
    assert np.all(adv == 0) and np.all(ret == 0)


# ---------------------------------------------------------------------------
# value loss and explained variance
# ---------------------------------------------------------------------------

def test_value_loss_zero_at_target():
    r = _rng(50)
    v = r.normal(size=20)
    m = (r.random(20) < 0.7).astype(np.uint8)
    loss, g, ev = O.value_loss(v, v, m)
    assert loss == 0.0 and np.all(g == 0.0)
    assert O.explained_variance(ev, int(m.sum())) == 1.0


def test_value_loss_finite_differences_and_mean():
    r = _rng(51)
    v = r.normal(size=15)
    R = r.normal(size=15)
    m = (r.random(15) < 0.6).astype(np.uint8)
    loss, g, _ = O.value_loss(v, R, m)
    mb = m.astype(bool)
    assert abs(loss - np.mean((v[mb] - R[mb]) ** 2)) < 1e-14
    for t in range(15):
        a = v.copy()
        a[t] += 1e-6
        b = v.copy()
        b[t] -= 1e-6
        num = (O.value_loss(a, R, m)[0] - O.value_loss(b, R, m)[0]) / 2e-6
        assert abs(num - g[t]) < 1e-8


def test_value_loss_external_normaliser_scales_loss_and_grad():
    # a batch split in two with the whole batch's count as the normaliser:
    # the halves' losses and gradients are the whole batch's, split
    r = _rng(53)
    v = r.normal(size=30)
    R = r.normal(size=30)
    m = (r.random(30) < 0.7).astype(np.uint8)
    n = int(m.sum())
    loss, g, _ = O.value_loss(v, R, m)
    l1, g1, _ = O.value_loss(v[:11], R[:11], m[:11], n_norm=n)
    l2, g2, _ = O.value_loss(v[11:], R[11:], m[11:], n_norm=n)
    assert abs(l1 + l2 - loss) < 1e-14
    assert np.array_equal(np.concatenate([g1, g2]), g)
    l3, g3, _ = O.value_loss(v, R, m, n_norm=4 * n)
    assert abs(4 * l3 - loss) < 1e-14 and np.allclose(4 * g3, g, rtol=1e-15, atol=0)


def test_explained_variance_matches_numpy_var():
    r = _rng(52)
    v = r.normal(size=100)
    R = v + r.normal(0, 0.3, size=100)
    m = (r.random(100) < 0.8).astype(np.uint8)
    _, _, ev = O.value_loss(v, R, m)
    mb = m.astype(bool)
    want = 1.0 - np.var(R[mb] - v[mb]) / np.var(R[mb])
    assert abs(O.explained_variance(ev, int(mb.sum())) - want) < 1e-12


# ---------------------------------------------------------------------------
# step-level GAE (App. A.1)
# ---------------------------------------------------------------------------

def test_step_gae_single_token_steps_equal_token_gae():
    """When every step is one action token (observations between them), both
    step values are the token value and step GAE is token GAE."""
    r = _rng(60)
    L = 41
    m = np.zeros(L, np.uint8)
    m[::2] = 1
    v = r.normal(0.4, 0.2, size=L)
    for mode in (O.STEP_AVERAGE, O.STEP_LAST):
        a_s, r_s, vm = O.step_advantages(v, np.array([1.0]), m, np.array([0, L]), 0.97, 0.9, 1.0, 1.5, mode)
        a_t, r_t = O.advantages(v, np.array([1.0]), m, np.array([0, L]), 0.97, 0.9, 1.0, 1.5)
        assert np.allclose(a_s, a_t, atol=1e-14) and np.allclose(r_s, r_t, atol=1e-14)
        assert np.array_equal(vm, m)


def test_step_gae_telescopes_and_broadcasts():
    """gamma = lambda = 1: every token of step i gets R - V(S_i); mean vs last."""
    m = np.array([0, 1, 1, 1, 0, 0, 1, 1, 0, 1], np.uint8)
    v = np.array([9.0, 0.1, 0.2, 0.6, 9.0, 9.0, 0.3, 0.5, 9.0, 0.7])
    R = 1.0
    a_avg, r_avg, vm_avg = O.step_advantages(v, np.array([R]), m, np.array([0, 10]), 1.0, 1.0, 1.0, 0.0,
                                             O.STEP_AVERAGE)
    assert np.allclose(a_avg[[1, 2, 3]], R - 0.3) and np.allclose(a_avg[[6, 7]], R - 0.4)
    assert np.allclose(a_avg[9], R - 0.7) and np.all(a_avg[m == 0] == 0)
    assert np.allclose(r_avg[m == 1], R) and np.array_equal(vm_avg, m)
    a_last, _, vm_last = O.step_advantages(v, np.array([R]), m, np.array([0, 10]), 1.0, 1.0, 1.0, 0.0,
                                           O.STEP_LAST)
    assert np.allclose(a_last[[1, 2, 3]], R - 0.6) and np.allclose(a_last[[6, 7]], R - 0.5)
    assert list(np.flatnonzero(vm_last)) == [3, 7, 9]


def test_step_gae_steps_stop_at_trajectory_ends():
    """Action runs that touch across a trajectory boundary are two steps, one
    per trajectory, each with its own reward; an empty trajectory and one with
    only observation tokens get nothing. gamma = lambda = 1: a step's
    advantage is its trajectory's reward minus the step value."""
    m = np.array([1, 1, 1, 1, 1, 0, 0], np.uint8)
    v = np.array([0.2, 0.4, 0.1, 0.3, 0.5, 9.0, 9.0])
    cu = np.array([0, 2, 2, 5, 7])                     # [0,2) | empty | [2,5) | [5,7) observations
    R = np.array([1.0, 7.0, 0.0, 3.0])
    a, r, vm = O.step_advantages(v, R, m, cu, 1.0, 1.0, 1.0, 0.0, O.STEP_AVERAGE)
    assert np.allclose(a[:2], 1.0 - 0.3) and np.allclose(a[2:5], 0.0 - 0.3)
    assert np.all(a[5:] == 0) and np.all(r[5:] == 0) and np.array_equal(vm, m)
    a, _, vm = O.step_advantages(v, R, m, cu, 1.0, 1.0, 1.0, 0.0, O.STEP_LAST)
    assert np.allclose(a[:2], 1.0 - 0.4) and np.allclose(a[2:5], 0.0 - 0.5)
    assert list(np.flatnonzero(vm)) == [1, 4]


def test_step_gae_explicit_sum_and_step_count_lambda():
    """Step advantages follow the explicit GAE sum over steps, with the
    length-adaptive lambda counted in steps (App. A.1)."""
    r = _rng(61)
    m = np.array([1, 1, 0, 1, 1, 1, 0, 0, 1, 0, 1, 1], np.uint8)
    v = r.normal(0.4, 0.2, size=len(m))
    a, _, _ = O.step_advantages(v, np.array([1.0]), m, np.array([0, len(m)]), 0.9, 0.5, 1.0, 1.5,
                                O.STEP_AVERAGE)
    vs = np.array([v[0:2].mean(), v[3:6].mean(), v[8], v[10:12].mean()])
    lam = 1.0 - 1.0 / (1.5 * 4)
    want = _explicit_sum_gae(vs, 1.0, 0.9, lam)
    assert np.allclose(a[[0, 3, 8, 10]], want, atol=1e-14)


# ---------------------------------------------------------------------------
# clipped surrogate (PPO / GRPO arms) and GRPO advantages
# ---------------------------------------------------------------------------

def test_clip_loss_no_bounds_equals_dis_without_bounds():
    logp, old, adv, m = _loss_inputs(70)
    cu = np.array([0, len(m)])
    a = O.clip_loss(logp, old, adv, m, cu, 1e30, 1e30, O.NORM_TOKEN)
    b = O.policy_loss(logp, old, adv, m, 1e30, 1e30)
    assert abs(a["loss"] - b["loss"]) < 1e-12 and np.allclose(a["coef"], b["coef"], atol=1e-15)


def test_clip_loss_clipping_is_strict_and_sign_dependent():
    """A ratio exactly at a bound gives min(rA, clip(r)A) = rA with both terms
    equal: not counted as clipped; one representable step outward is. A ratio
    above 1+eps_high with A < 0 (or below 1-eps_low with A > 0) is never
    clipped: the min takes the unclipped term."""
    for d in (np.float32(0.25), np.float32(0.6)):
        r = np.float32(np.exp(d))
        eps_h = float(r - np.float32(1.0))                # exact (Sterbenz)
        assert np.float32(1.0) + np.float32(eps_h) == r
        assert O.clip_flags([d], [0.0], [1.0], [1], 0.5, eps_h)[0] == O.CLIP_NONE
        d_out = np.nextafter(d, np.float32(1.0))
        if np.float32(np.exp(d_out)) > r:
            assert O.clip_flags([d_out], [0.0], [1.0], [1], 0.5, eps_h)[0] == O.CLIP_HIGH
        assert O.clip_flags([d_out], [0.0], [-1.0], [1], 0.5, eps_h)[0] == O.CLIP_NONE
    for d in (np.float32(-0.25), np.float32(-0.6)):
        r = np.float32(np.exp(d))
        eps_l = float(np.float32(1.0) - r)
        assert np.float32(1.0) - np.float32(eps_l) == r
        assert O.clip_flags([d], [0.0], [-1.0], [1], eps_l, 0.5)[0] == O.CLIP_NONE
        d_out = np.nextafter(d, np.float32(-1.0))
        if np.float32(np.exp(d_out)) < r:
            assert O.clip_flags([d_out], [0.0], [-1.0], [1], eps_l, 0.5)[0] == O.CLIP_LOW
        assert O.clip_flags([d_out], [0.0], [1.0], [1], eps_l, 0.5)[0] == O.CLIP_NONE


def test_clip_loss_hand_example():
    """A > 0 above 1+eps_high and A < 0 below 1-eps_low are clipped (value at the
    bound, zero gradient); A > 0 below 1-eps_low and A < 0 above 1+eps_high are
    not (the min keeps r*A)."""
    logp = np.log(np.array([1.5, 0.5, 0.5, 1.5, 1.0])).astype(np.float32)
    old = np.zeros(5, np.float32)
    adv = np.array([2.0, -1.0, 1.0, -0.5, 0.25], np.float32)
    m = np.ones(5, np.uint8)
    out = O.clip_loss(logp, old, adv, m, np.array([0, 5]), 0.2, 0.28, O.NORM_TOKEN)
    assert list(out["flags"]) == [2, 1, 0, 0, 0]
    r = np.exp(logp.astype(np.float64))
    lo, hi = float(np.float32(0.8)), float(np.float32(1.0) + np.float32(0.28))
    want = -(hi * 2.0 + lo * -1.0 + r[2] * 1.0 + r[3] * -0.5 + r[4] * 0.25) / 5
    assert abs(out["loss"] - want) < 1e-12
    assert out["coef"][0] == 0 and out["coef"][1] == 0
    assert abs(out["coef"][3] - (-(r[3] * -0.5) / 5)) < 1e-15


def test_clip_loss_sequence_normalisation():
    """Sequence mode: each trajectory's tokens average first, so a 1-token
    trajectory weighs as much as a 3-token one; old = new gives minus the mean
    over trajectories of the per-trajectory mean advantage."""
    adv = np.array([1.0, 2.0, 3.0, 10.0], np.float32)
    lp = np.full(4, -1.0, np.float32)
    m = np.ones(4, np.uint8)
    cu = np.array([0, 3, 4])
    out = O.clip_loss(lp, lp, adv, m, cu, 0.2, 0.28, O.NORM_SEQUENCE)
    assert abs(out["loss"] - (-(2.0 + 10.0) / 2)) < 1e-12
    tok = O.clip_loss(lp, lp, adv, m, cu, 0.2, 0.28, O.NORM_TOKEN)
    assert abs(tok["loss"] - (-16.0 / 4)) < 1e-12


def test_clip_loss_finite_differences():
    logp, old, adv, m = _loss_inputs(71, N=20)
    cu = np.array([0, 7, 7, 20])
    for norm in (O.NORM_TOKEN, O.NORM_SEQUENCE):
        out = O.clip_loss(logp, old, adv, m, cu, 0.2, 0.28, norm)
        lp = logp.astype(np.float64)
        for t in range(20):
            r = math.exp(lp[t] - float(old[t]))
            if abs(r - 0.8) < 1e-4 or abs(r - 1.28) < 1e-4:
                continue
            a, b = lp.copy(), lp.copy()
            a[t] += 1e-7
            b[t] -= 1e-7
            num = (O.clip_loss(a, old, adv, m, cu, 0.2, 0.28, norm)["loss"] -
                   O.clip_loss(b, old, adv, m, cu, 0.2, 0.28, norm)["loss"]) / 2e-7
            assert abs(num - out["coef"][t]) < 1e-7


def test_group_advantages_are_standardised():
    r = _rng(72)
    B = 24
    gid = np.repeat(np.arange(3), 8)
    R = (r.random(B) < 0.5).astype(np.float32)
    R[16:] = 1.0                                       # a constant group
    lens = r.integers(1, 9, size=B)
    cu = np.concatenate([[0], np.cumsum(lens)])
    m = np.ones(cu[-1], np.uint8)
    adv = O.group_advantages(R, gid, m, cu, 1e-6)
    per_traj = adv[cu[:-1]]
    for g in range(2):
        a = per_traj[gid == g]
        var = np.var(R[gid == g].astype(np.float64))
        assert abs(a.mean()) < 1e-12
        assert abs(np.mean(a ** 2) - var / (var + 1e-6)) < 1e-9
    assert np.all(per_traj[gid == 2] == 0)
    single = O.group_advantages(np.array([1.0], np.float32), np.array([0]), np.ones(3, np.uint8),
                                np.array([0, 3]), 1e-6)
    assert np.all(single == 0)


def test_group_advantages_two_members_closed_form():
    """A group {0, 1} interleaved with another in the batch, eps 0: population
    variance 1/4, so the advantages are exactly -1 and +1 (a sample variance
    would give -/+ 1/sqrt(2)); observation tokens get 0. A group of equal
    rewards gets 0 once eps > 0 (with eps 0 it is 0/0: eps sits under the
    square root for this case)."""
    R = np.array([0.0, 3.0, 1.0, 5.0], np.float32)
    gid = np.array([7, 9, 7, 9])
    cu = np.array([0, 3, 5, 9, 10])
    m = np.array([1, 0, 1, 1, 1, 0, 1, 1, 0, 1], np.uint8)
    adv = O.group_advantages(R, gid, m, cu, 0.0)
    want = np.array([-1, 0, -1, -1, -1, 0, 1, 1, 0, 1], np.float64)
    assert np.array_equal(adv, want)
    R[3] = 3.0
    adv = O.group_advantages(R, gid, m, cu, 1e-6)
    assert np.all(adv[3:5] == 0) and adv[9] == 0


def test_running_mean_window_one_and_ring_wrap():
    """Window 1: the baseline is the prompt's previous reward. Window 3 over
    rewards 1..7 of one prompt: the baseline of reward k is the mean of the
    (up to) three before it, across two batches, with the ring wrapping."""
    R = np.array([2.0, 5.0, 1.0], np.float32)
    pid = np.zeros(3, np.int64)
    cu = np.arange(4)
    m = np.ones(3, np.uint8)
    adv, _, _ = O.running_mean_advantages(R, pid, m, cu, np.zeros((1, 1)), np.zeros(1, np.int64), 1)
    assert np.allclose(adv, [2.0, 3.0, -4.0])
    hist, seen = np.zeros((1, 3)), np.zeros(1, np.int64)
    got = []
    for batch in (np.arange(1, 5), np.arange(5, 8)):
        a, hist, seen = O.running_mean_advantages(batch.astype(np.float32), np.zeros(len(batch), np.int64),
                                                  np.ones(len(batch), np.uint8), np.arange(len(batch) + 1),
                                                  hist, seen, 3)
        got.extend(a)
    want = [1.0, 2.0 - 1.0, 3.0 - 1.5, 4.0 - 2.0, 5.0 - 3.0, 6.0 - 4.0, 7.0 - 5.0]
    assert np.allclose(got, want) and int(seen[0]) == 7


def test_running_mean_baseline_window():
    """Window 2 for prompt 0 over rewards 1, 0, 1, 1: baselines 0 (empty), 1,
    mean(1, 0), mean(0, 1); prompt 1 keeps its own window."""
    R = np.array([1.0, 0.0, 1.0, 5.0, 1.0], np.float32)
    pid = np.array([0, 0, 0, 1, 0])
    cu = np.arange(6)
    m = np.ones(5, np.uint8)
    adv, hist, cnt = O.running_mean_advantages(R, pid, m, cu, np.zeros((2, 2)), np.zeros(2, np.int64), 2)
    assert np.allclose(adv, [1.0, -1.0, 0.5, 5.0, 0.5])
    assert list(cnt) == [4, 1] and sorted(hist[0]) == [1.0, 1.0] and hist[1, 0] == 5.0
    # the state carries over to the next batch
    adv2, _, _ = O.running_mean_advantages(np.array([0.0], np.float32), np.array([0]), np.ones(1, np.uint8),
                                           np.array([0, 1]), hist, cnt, 2)
    assert np.allclose(adv2, [-1.0])


# ---------------------------------------------------------------------------
# decoupled three-policy objective (§3.1), reading R17
# ---------------------------------------------------------------------------

def _three_policies(seed, N=200):
    r = _rng(seed)
    logp = (-r.exponential(2.0, N)).astype(np.float32)
    prox = (logp + r.normal(0, 0.2, N)).astype(np.float32)
    roll = (prox + r.normal(0, 0.3, N)).astype(np.float32)
    adv = r.normal(size=N).astype(np.float32)
    m = (r.random(N) < 0.8).astype(np.uint8)
    return logp, prox, roll, adv, m


def test_decoupled_loss_equal_old_and_rollout_is_the_clipped_surrogate():
    """pi_old = pi_rollout makes the mismatch weight 1 (inside the band): the
    objective is the token-mean clipped surrogate against pi_old."""
    logp, prox, _, adv, m = _three_policies(80)
    d = O.decoupled_loss(logp, prox, prox, adv, m, 0.2, 0.28, 0.5, 2.0)
    c = O.clip_loss(logp, prox, adv, m, np.array([0, len(m)]), 0.2, 0.28, O.NORM_TOKEN)
    assert abs(d["loss"] - c["loss"]) < 1e-12
    assert np.allclose(d["coef"], c["coef"], atol=1e-15) and np.array_equal(d["flags"], c["flags"])
    assert list(d["counts"][:4]) == list(c["counts"]) and d["counts"][4] == d["counts"][5] == 0


def test_decoupled_loss_without_bounds_telescopes_to_eq1():
    """With every bound off, w*r = pi_theta/pi_rollout: the loss is Eq. 1 with
    f = identity against the rollout log-probs, -(1/n) sum exp(logp - rollout) A."""
    logp, prox, roll, adv, m = _three_policies(81)
    d = O.decoupled_loss(logp, prox, roll, adv, m, 1e30, 1e30, 0.0, np.inf)
    k = m.astype(bool)
    lp, ro, a = (x.astype(np.float64) for x in (logp, roll, adv))
    want = -math.fsum(np.exp(lp[k] - ro[k]) * a[k]) / k.sum()
    assert abs(d["loss"] - want) < 1e-12
    dis = O.policy_loss(logp, roll, adv, m, 1e30, 1e30)
    assert np.allclose(d["coef"], dis["coef"], atol=1e-15)


def test_decoupled_loss_hand_example():
    """Token 0: w = 2.5 >= 2 (masked high); 1: w = 0.25 <= 0.5 (masked low);
    2: w = 1.25 kept, r = 1.5 > 1.28 with A > 0 (clipped: w*(1+eps_high)*A, no
    gradient); 3: w = 1, r = 0.9 with A < 0 above 1-eps_low (unclipped: w*r*A);
    4: not an action token."""
    logp = np.log(np.array([1.0, 1.0, 1.5, 0.9, 1.0])).astype(np.float32)
    prox = np.zeros(5, np.float32)
    roll = np.log(np.array([0.4, 4.0, 0.8, 1.0, 1.0])).astype(np.float32)
    adv = np.array([1.0, 1.0, 2.0, -1.0, 3.0], np.float32)
    m = np.array([1, 1, 1, 1, 0], np.uint8)
    out = O.decoupled_loss(logp, prox, roll, adv, m, 0.2, 0.28, 0.5, 2.0)
    assert list(out["flags"]) == [O.MIS_HIGH, O.MIS_LOW, O.CLIP_HIGH, O.CLIP_NONE, O.FLAG_MASKED]
    assert list(out["counts"]) == [4, 0, 1, 0, 1, 1]
    w2 = math.exp(-float(roll[2]))
    r3 = math.exp(float(logp[3]))
    hi = float(np.float32(1.0) + np.float32(0.28))
    assert abs(out["loss"] - (-(w2 * hi * 2.0 + 1.0 * r3 * -1.0) / 4)) < 1e-12
    assert out["coef"][2] == 0 and abs(out["coef"][3] - (r3 / 4)) < 1e-15


def test_decoupled_loss_band_is_strict():
    """w = 1 exactly (pi_old = pi_rollout): masked when a band edge equals 1."""
    lp = np.zeros(3, np.float32)
    adv = np.ones(3, np.float32)
    m = np.ones(3, np.uint8)
    assert set(O.decoupled_loss(lp, lp, lp, adv, m, 0.2, 0.28, 1.0, 2.0)["flags"]) == {O.MIS_LOW}
    assert set(O.decoupled_loss(lp, lp, lp, adv, m, 0.2, 0.28, 0.5, 1.0)["flags"]) == {O.MIS_HIGH}
    assert set(O.decoupled_loss(lp, lp, lp, adv, m, 0.2, 0.28, 0.5, 2.0)["flags"]) == {O.CLIP_NONE}


def test_decoupled_loss_finite_differences_and_normaliser():
    logp, prox, roll, adv, m = _three_policies(82, N=24)
    out = O.decoupled_loss(logp, prox, roll, adv, m, 0.2, 0.28, 0.5, 2.0, n_norm=7)
    lp = logp.astype(np.float64)
    for t in range(24):
        r = math.exp(lp[t] - float(prox[t]))
        if abs(r - 0.8) < 1e-4 or abs(r - 1.28) < 1e-4:
            continue
        a, b = lp.copy(), lp.copy()
        a[t] += 1e-7
        b[t] -= 1e-7
        num = (O.decoupled_loss(a, prox, roll, adv, m, 0.2, 0.28, 0.5, 2.0, n_norm=7)["loss"] -
               O.decoupled_loss(b, prox, roll, adv, m, 0.2, 0.28, 0.5, 2.0, n_norm=7)["loss"]) / 2e-7
        assert abs(num - out["coef"][t]) < 1e-7


def test_decoupled_loss_nonfinite_tokens_are_masked():
    logp, prox, roll, adv, m = _three_policies(83, N=30)
    m[:] = 1
    roll[3] = -np.inf
    prox[5] = np.nan
    adv[7] = np.inf
    out = O.decoupled_loss(logp, prox, roll, adv, m, 0.2, 0.28, 0.5, 2.0)
    assert all(out["flags"][t] == O.FLAG_NONFINITE for t in (3, 5, 7))
    assert out["counts"][3] == 3 and out["counts"][0] == 30 and np.isfinite(out["loss"])


# ---------------------------------------------------------------------------
# helpers the entry points build on, pinned directly
# ---------------------------------------------------------------------------

def test_trajectory_lambda_hand_values():
    # lambda = 1 - 1/(alpha * l), clamped to [0, 1]; alpha <= 0 keeps the fixed lambda (§4.1)
    assert O.trajectory_lambda(0.95, 0.0, 10) == 0.95
    assert abs(O.trajectory_lambda(0.95, 1.5, 3) - (1.0 - 1.0 / 4.5)) < 1e-15
    assert O.trajectory_lambda(0.95, 1.5, 0) == 0.0
    assert O.trajectory_lambda(0.95, 0.5, 1) == 0.0          # 1 - 1/0.5 < 0
    assert abs(O.trajectory_lambda(0.95, 1.5, 128_000) - (1.0 - 1.0 / 192_000)) < 1e-15


def test_step_spans_hand_cases():
    m = np.array([1, 1, 0, 1, 0, 0, 1, 1, 1], np.uint8)
    assert O.step_spans(m, 0, 9) == [(0, 2), (3, 4), (6, 9)]
    assert O.step_spans(m, 1, 7) == [(1, 2), (3, 4), (6, 7)]   # clipped at the trajectory's bounds
    assert O.step_spans(np.zeros(5, np.uint8), 0, 5) == []
    assert O.step_spans(np.ones(4, np.uint8), 0, 4) == [(0, 4)]


def test_decoupled_flags_hand_cases():
    # r = pi_theta / pi_old, w = pi_old / pi_rollout; band (w_low, w_high) = (0.5, 2.0), eps 0.2 / 0.28
    ln = np.log
    logp = np.array([0.0, ln(1.5), ln(0.5), 0.0, 0.0, 0.0, np.nan, 0.0], np.float32)
    prox = np.zeros(8, np.float32)
    roll = np.array([0.0, 0.0, 0.0, ln(4.0), -ln(3.0), 0.0, 0.0, 0.0], np.float32)
    adv = np.array([1.0, 1.0, -1.0, 1.0, 1.0, -1.0, 1.0, 1.0], np.float32)
    m = np.array([1, 1, 1, 1, 1, 1, 1, 0], np.uint8)
    f = O.decoupled_flags(logp, prox, roll, adv, m, 0.2, 0.28, 0.5, 2.0)
    # kept; r = 1.5 > 1.28 with A > 0: clip high; r = 0.5 < 0.8 with A < 0: clip low;
    # w = 1/4 <= 0.5: mismatch low; w = 3 >= 2: mismatch high; kept (A < 0, r = 1);
    # non-finite log-ratio; not an action token
    assert list(f) == [0, 2, 1, 5, 6, 0, 3, 4]
