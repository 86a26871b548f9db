"""GPU parity of the follow-on rows (the paper's variants and comparison
arms) with the fp64 oracle, through the C ABI."""
import numpy as np
import pytest
import torch

from oracle import sao_oracle as O
from paper_2607_07508_gb300 import sao, synthetic as S
from tests._util import cuda, rel_err_floor

pytestmark = pytest.mark.gpu

ADV_TOL = 1e-5


def f32(x):
    return float(np.float32(x))


def _step_gpu(wl, gamma, lam, lam_c, alpha, mode):
    N = wl.N
    adv = torch.full((N,), float("nan"), device="cuda")
    ret = torch.full((N,), float("nan"), device="cuda")
    vm = torch.full((N,), 7, dtype=torch.uint8, device="cuda")
    sao.sao_step_advantages(cuda(wl.values), cuda(wl.rewards), cuda(wl.loss_mask), cuda(wl.cu_seqlens), gamma,
                            lam, lam_c, alpha, mode, adv, ret, sao.workspace(N), value_mask=vm)
    torch.cuda.synchronize()
    return adv.cpu().numpy(), ret.cpu().numpy(), vm.cpu().numpy()


def _check_step(wl, gamma, lam, lam_c, alpha, mode):
    gamma, lam, lam_c, alpha = f32(gamma), f32(lam), f32(lam_c), f32(alpha)
    adv, ret, vm = _step_gpu(wl, gamma, lam, lam_c, alpha, mode)
    wa, wr, wv = O.step_advantages(wl.values, wl.rewards, wl.loss_mask, wl.cu_seqlens, gamma, lam, lam_c, alpha,
                                   mode)
    assert rel_err_floor(adv, wa, 1e-3).max() <= ADV_TOL
    assert rel_err_floor(ret, wr, 1e-3).max() <= ADV_TOL
    assert np.array_equal(vm, wv)


@pytest.mark.parametrize("mode", [sao.SAO_STEP_AVERAGE, sao.SAO_STEP_LAST])
@pytest.mark.parametrize("name", S.CONFIG_NAMES)
def test_step_advantages_match_oracle(name, mode):
    wl = S.make_workload(name, dense=False)
    _check_step(wl, wl.gamma, wl.lam, wl.lam_critic, wl.alpha, mode)


@pytest.mark.parametrize("mode", [sao.SAO_STEP_AVERAGE, sao.SAO_STEP_LAST])
@pytest.mark.parametrize("lengths", [[1], [5, 0, 0, 7], [0, 4096, 1, 4095, 0], [3] * 500, [70001]])
def test_step_advantages_edge_layouts(lengths, mode):
    wl = S.make_custom(lengths, 8, 16, "f32", seed=sum(lengths) + 3, dense=False, obs_frac=0.4)
    wl.loss_mask[::31] = 0
    _check_step(wl, 0.99, 0.95, 0.97, 1.5, mode)
    _check_step(wl, 1.0, 0.9, 1.0, 0.0, mode)


def test_step_advantages_misaligned_outputs():
    """Outputs and inputs one element past a 16-byte boundary: the scalar paths
    of the count, scatter and broadcast passes give the same results."""
    wl = S.make_custom([3, 0, 4100, 1, 900], 8, 16, "f32", seed=21, dense=False, obs_frac=0.4)
    N = wl.N
    mis = lambda t: torch.cat([t[:1], t])[1:]
    adv = mis(torch.full((N,), float("nan"), device="cuda"))
    ret = mis(torch.full((N,), float("nan"), device="cuda"))
    vm = mis(torch.full((N,), 7, dtype=torch.uint8, device="cuda"))
    for mode in (sao.SAO_STEP_AVERAGE, sao.SAO_STEP_LAST):
        sao.sao_step_advantages(mis(cuda(wl.values)), cuda(wl.rewards), mis(cuda(wl.loss_mask)), cuda(wl.cu_seqlens),
                                1.0, f32(0.95), 1.0, 0.0, mode, adv, ret, sao.workspace(N), value_mask=vm)
        torch.cuda.synchronize()
        wa, wr, wv = O.step_advantages(wl.values, wl.rewards, wl.loss_mask, wl.cu_seqlens, 1.0, f32(0.95), 1.0, 0.0,
                                       mode)
        assert rel_err_floor(adv.cpu().numpy(), wa, 1e-3).max() <= ADV_TOL
        assert rel_err_floor(ret.cpu().numpy(), wr, 1e-3).max() <= ADV_TOL
        assert np.array_equal(vm.cpu().numpy(), wv)


@pytest.mark.parametrize("mode", [sao.SAO_STEP_AVERAGE, sao.SAO_STEP_LAST])
def test_step_advantages_large_batch(mode):
    """2^25 + 4,321 tokens of turn-length steps: from 2^25 tokens the per-step
    sums take 32 steps per warp, and the broadcast's groups are not split; 48
    sampled trajectories and the last two (the ragged tail) against the oracle
    on their own slices."""
    N = (1 << 25) + 4321
    wl = S.bandwidth_workload(N=N, B=max(1, N >> 13))
    g, lam, lc, al = f32(0.99), f32(0.95), f32(0.97), f32(1.5)
    adv, ret, vm = _step_gpu(wl, g, lam, lc, al, mode)
    rng = np.random.default_rng(mode + 5)
    picks = np.concatenate([rng.choice(wl.B, size=48, replace=False), [wl.B - 2, wl.B - 1]])
    for b in picks:
        lo, hi = wl.cu_seqlens[b], wl.cu_seqlens[b + 1]
        wa, wr, wv = O.step_advantages(wl.values[lo:hi], wl.rewards[b:b + 1], wl.loss_mask[lo:hi],
                                       np.array([0, hi - lo]), g, lam, lc, al, mode)
        assert rel_err_floor(adv[lo:hi], wa, 1e-3).max() <= ADV_TOL
        assert rel_err_floor(ret[lo:hi], wr, 1e-3).max() <= ADV_TOL
        assert np.array_equal(vm[lo:hi], wv)


@pytest.mark.parametrize("N", [(1 << 20) + 3, (1 << 25) + 777])
def test_step_advantages_short_steps(N):
    """Token-by-token random masks: steps of 1-3 tokens, several inside one
    lane's 4 tokens (the broadcast's per-token search), one lane per short step
    in the per-step sums, millions of steps; sampled trajectories and the
    ragged tail against the oracle on their own slices, both value modes."""
    wl = S.bandwidth_workload(N=N, B=max(1, N >> 13))
    rng = np.random.default_rng(N % 997)
    wl.loss_mask = (rng.random(N) < 0.6).astype(np.uint8)
    g, lam, lc = f32(1.0), f32(0.95), f32(1.0)
    picks = np.concatenate([rng.choice(wl.B, size=24, replace=False), [wl.B - 2, wl.B - 1]])
    for mode in (sao.SAO_STEP_AVERAGE, sao.SAO_STEP_LAST):
        adv, ret, vm = _step_gpu(wl, g, lam, lc, 0.0, mode)
        for b in picks:
            lo, hi = wl.cu_seqlens[b], wl.cu_seqlens[b + 1]
            wa, wr, wv = O.step_advantages(wl.values[lo:hi], wl.rewards[b:b + 1], wl.loss_mask[lo:hi],
                                           np.array([0, hi - lo]), g, lam, lc, 0.0, mode)
            assert rel_err_floor(adv[lo:hi], wa, 1e-3).max() <= ADV_TOL
            assert rel_err_floor(ret[lo:hi], wr, 1e-3).max() <= ADV_TOL
            assert np.array_equal(vm[lo:hi], wv)


def test_step_advantages_no_action_tokens():
    wl = S.make_custom([10, 300], 8, 16, "f32", seed=4, dense=False)
    wl.loss_mask[:] = 0
    adv, ret, vm = _step_gpu(wl, 1.0, 1.0, 1.0, 0.0, sao.SAO_STEP_AVERAGE)
    assert not adv.any() and not ret.any() and not vm.any()


# ---------------------------------------------------------------------------
# clipped surrogate (PPO / GRPO arms) and GRPO advantages
# ---------------------------------------------------------------------------

def _clip_gpu(logp, old, adv, mask, cu, el, eh, norm):
    N = len(logp)
    loss = torch.empty(1, device="cuda")
    counts = torch.empty(4, dtype=torch.int64, device="cuda")
    coef = torch.empty(N, device="cuda")
    flags = torch.empty(N, dtype=torch.uint8, device="cuda")
    grad = torch.empty(N, device="cuda")
    ws = sao.workspace(N)
    args = [cuda(x) for x in (logp, old, adv, mask, cu)]
    sao.sao_clip_loss_fwd(*args, el, eh, norm, loss, counts, ws, coef=coef, flags=flags)
    sao.sao_clip_loss_bwd(*args, el, eh, norm, torch.tensor([0.5], device="cuda"), grad, ws)
    torch.cuda.synchronize()
    return float(loss.item()), counts.cpu().numpy(), coef.cpu().numpy(), flags.cpu().numpy(), grad.cpu().numpy()


def _near_clip_bound(logp, old, el, eh, tol=1e-6):
    r = np.exp(np.asarray(logp, np.float64) - np.asarray(old, np.float64))
    with np.errstate(invalid="ignore"):
        return (np.abs(r - (1 - el)) <= tol) | (np.abs(r - (1 + eh)) <= tol)


@pytest.mark.parametrize("norm", [sao.SAO_NORM_TOKEN, sao.SAO_NORM_SEQUENCE])
@pytest.mark.parametrize("name", S.CONFIG_NAMES)
def test_clip_loss_match_oracle(name, norm):
    wl = S.make_workload(name, dense=False)
    adv = np.random.default_rng(5).normal(size=wl.N).astype(np.float32)
    el, eh = 0.2, 0.28
    loss, counts, coef, flags, grad = _clip_gpu(wl.logp_syn, wl.old_logp_syn, adv, wl.loss_mask, wl.cu_seqlens,
                                                el, eh, norm)
    want = O.clip_loss(wl.logp_syn, wl.old_logp_syn, adv, wl.loss_mask, wl.cu_seqlens, el, eh, norm)
    skip = _near_clip_bound(wl.logp_syn, wl.old_logp_syn, el, eh)
    assert np.array_equal(flags[~skip], want["flags"][~skip])
    if not skip.any():
        assert np.array_equal(counts, want["counts"])
    assert abs(loss - want["loss"]) <= 1e-4 * max(abs(want["loss"]), 1e-6)
    keep = ~skip
    assert rel_err_floor(coef[keep], want["coef"][keep], 1e-12).max() <= 1e-5
    assert rel_err_floor(grad[keep], 0.5 * want["coef"][keep], 1e-12).max() <= 1e-5


@pytest.mark.parametrize("norm", [sao.SAO_NORM_TOKEN, sao.SAO_NORM_SEQUENCE])
def test_clip_loss_edge_layouts(norm):
    wl = S.make_custom([0, 1, 1023, 0, 2049, 5], 8, 16, "f32", seed=8, dense=False, obs_frac=0.3)
    rng = np.random.default_rng(6)
    adv = rng.normal(size=wl.N).astype(np.float32)
    old = (wl.logp_syn + rng.normal(0, 0.5, wl.N)).astype(np.float32)
    old[::50] = -np.inf
    loss, counts, coef, flags, grad = _clip_gpu(wl.logp_syn, old, adv, wl.loss_mask, wl.cu_seqlens, 0.3, 5.0, norm)
    want = O.clip_loss(wl.logp_syn, old, adv, wl.loss_mask, wl.cu_seqlens, 0.3, 5.0, norm)
    assert np.array_equal(flags, want["flags"]) and np.array_equal(counts, want["counts"])
    assert abs(loss - want["loss"]) <= 1e-4 * max(abs(want["loss"]), 1e-6)
    assert rel_err_floor(coef, want["coef"], 1e-12).max() <= 1e-5



@pytest.mark.parametrize("norm", [sao.SAO_NORM_TOKEN, sao.SAO_NORM_SEQUENCE])
def test_clip_loss_short_trajectories_and_misaligned_inputs(norm):
    """Trajectories of 0 to 6 tokens (hundreds per 1024-token chunk, more than
    a chunk stages, so the walk reads the offsets from global memory) around
    two long ones and a ragged tail; once with aligned inputs (the staged
    path) and once with every input one element past a 16-byte boundary (the
    scalar path)."""
    rng = np.random.default_rng(12)
    lengths = [int(x) for x in rng.integers(0, 7, size=1500)]
    lengths[700] = 3000
    lengths[-2] = 1500
    wl = S.make_custom(lengths, 8, 16, "f32", seed=13, dense=False, obs_frac=0.3)
    adv = rng.normal(size=wl.N).astype(np.float32)
    old = (wl.logp_syn + rng.normal(0, 0.4, wl.N)).astype(np.float32)
    el, eh = 0.2, 0.28
    want = O.clip_loss(wl.logp_syn, old, adv, wl.loss_mask, wl.cu_seqlens, el, eh, norm)
    skip = _near_clip_bound(wl.logp_syn, old, el, eh)
    keep = ~skip
    for mis in (False, True):
        N = wl.N
        place = _misaligned if mis else (lambda t: t)
        loss = torch.empty(1, device="cuda")
        counts = torch.empty(4, dtype=torch.int64, device="cuda")
        coef = place(torch.full((N,), float("nan"), device="cuda"))
        flags = place(torch.full((N,), 9, dtype=torch.uint8, device="cuda"))
        grad = place(torch.full((N,), float("nan"), device="cuda"))
        ws = sao.workspace(N)
        args = [place(cuda(x)) for x in (wl.logp_syn, old, adv, wl.loss_mask)] + [cuda(wl.cu_seqlens)]
        sao.sao_clip_loss_fwd(*args, el, eh, norm, loss, counts, ws, coef=coef, flags=flags)
        sao.sao_clip_loss_bwd(*args, el, eh, norm, torch.tensor([2.0], device="cuda"), grad, ws)
        torch.cuda.synchronize()
        got_flags = flags.cpu().numpy()
        assert np.array_equal(got_flags[keep], want["flags"][keep]), mis
        if not skip.any():
            assert np.array_equal(counts.cpu().numpy(), want["counts"]), mis
        assert abs(loss.item() - want["loss"]) <= 1e-4 * max(abs(want["loss"]), 1e-6), mis
        assert rel_err_floor(coef.cpu().numpy()[keep], want["coef"][keep], 1e-12).max() <= 1e-5, mis
        assert rel_err_floor(grad.cpu().numpy()[keep], 2.0 * want["coef"][keep], 1e-12).max() <= 1e-5, mis

def test_group_advantages_match_oracle():
    for name in ("small", "large"):
        wl = S.make_workload(name, dense=False)
        gid = (np.arange(wl.B) // 8).astype(np.int32)            # 8 rollouts per prompt
        rng = np.random.default_rng(3)
        rng.shuffle(gid)
        adv = torch.empty(wl.N, device="cuda")
        sao.sao_group_advantages(cuda(wl.rewards), cuda(gid), cuda(wl.loss_mask), cuda(wl.cu_seqlens), 1e-6, adv,
                                 sao.workspace(wl.N))
        torch.cuda.synchronize()
        want = O.group_advantages(wl.rewards, gid, wl.loss_mask, wl.cu_seqlens, f32(1e-6))
        assert rel_err_floor(adv.cpu().numpy(), want, 1e-3).max() <= 1e-5


@pytest.mark.parametrize("seed", [0, 1])
def test_group_advantages_sorted_ids_same_bits(seed):
    """Non-decreasing group ids (a prompt's rollouts adjacent) take the path
    that visits only each CTA's runs: groups of 1 to 3,000 trajectories, runs
    across the 2,048-entry tiles, negative ids. Against the oracle, and bit
    for bit against the same partition under ids relabelled out of order
    (which takes the whole-batch scan)."""
    rng = np.random.default_rng(seed)
    sizes = np.concatenate([[1, 2, 3000, 8, 1], rng.integers(1, 60, size=300), [2500, 5]])
    B = int(sizes.sum())
    lengths = rng.integers(0, 40, size=B)
    wl = S.make_custom(lengths.tolist(), 8, 16, "f32", seed=21 + seed, dense=False, obs_frac=0.3)
    gid = (np.repeat(np.arange(len(sizes)), sizes) - 3).astype(np.int32)
    relabel = ((gid.astype(np.int64) + 3) * 7919 % 100003).astype(np.int32)
    assert np.any(np.diff(relabel) < 0) and np.all(np.diff(gid) >= 0)
    outs = []
    for ids in (gid, relabel):
        adv = torch.empty(wl.N, device="cuda")
        sao.sao_group_advantages(cuda(wl.rewards), cuda(ids), cuda(wl.loss_mask), cuda(wl.cu_seqlens), 1e-6, adv,
                                 sao.workspace(wl.N))
        torch.cuda.synchronize()
        outs.append(adv.cpu().numpy())
    assert np.array_equal(outs[0], outs[1])
    want = O.group_advantages(wl.rewards, gid, wl.loss_mask, wl.cu_seqlens, f32(1e-6))
    assert rel_err_floor(outs[0], want, 1e-3).max() <= 1e-5


def test_running_mean_advantages_match_oracle():
    """Two batches in a row with per-prompt windows of 8 (§4.3) and one global
    window of 128 (§4.5); the windows persist between calls."""
    for P, window in ((16, 8), (1, 128)):
        hist_d = torch.zeros(P, window, device="cuda")
        seen_d = torch.zeros(P, dtype=torch.int64, device="cuda")
        hist_o, seen_o = np.zeros((P, window)), np.zeros(P, np.int64)
        for seed in (1, 2):
            wl = S.make_workload("large", dense=False, seed=S.SEED_BASE + 40 + seed)
            pid = np.random.default_rng(seed).integers(0, P, size=wl.B).astype(np.int32)
            adv = torch.empty(wl.N, device="cuda")
            sao.sao_running_mean_advantages(cuda(wl.rewards), cuda(pid), hist_d, seen_d, cuda(wl.loss_mask),
                                            cuda(wl.cu_seqlens), adv, sao.workspace(wl.N))
            torch.cuda.synchronize()
            want, hist_o, seen_o = O.running_mean_advantages(wl.rewards, pid, wl.loss_mask, wl.cu_seqlens, hist_o,
                                                             seen_o, window)
            assert rel_err_floor(adv.cpu().numpy(), want, 1e-3).max() <= 1e-5
            assert np.array_equal(seen_d.cpu().numpy(), seen_o)
            assert np.allclose(hist_d.cpu().numpy(), hist_o)


def _misaligned(t):
    """The same values one element past a 16-byte boundary (scalar paths)."""
    pad = torch.empty(t.numel() + 1, dtype=t.dtype, device=t.device)
    pad[1:] = t
    return pad[1:]


def test_group_and_running_mean_edge_layouts():
    """5,003 trajectories (several shared-memory tiles, a partly filled last
    CTA), empty and one-token trajectories, ragged lengths, a misaligned mask
    and output (the broadcast's scalar path), and for the running mean two
    batches with per-prompt windows of 8, one window of 128, and 5,000 prompts
    (the walk without the rank table)."""
    rng = np.random.default_rng(11)
    lengths = rng.integers(0, 40, size=5003)
    lengths[:3] = [0, 1, 0]
    lengths[-2:] = [0, 1]
    wl = S.make_custom(lengths.tolist(), 8, 16, "f32", seed=12, dense=False, obs_frac=0.3)
    m_d, cu_d, R_d = _misaligned(cuda(wl.loss_mask)), cuda(wl.cu_seqlens), cuda(wl.rewards)
    gid = rng.integers(-5, 600, size=wl.B).astype(np.int32)
    adv = _misaligned(torch.full((wl.N,), float("nan"), device="cuda"))
    sao.sao_group_advantages(R_d, cuda(gid), m_d, cu_d, 1e-6, adv, sao.workspace(wl.N))
    torch.cuda.synchronize()
    want = O.group_advantages(wl.rewards, gid, wl.loss_mask, wl.cu_seqlens, f32(1e-6))
    assert rel_err_floor(adv.cpu().numpy(), want, 1e-3).max() <= 1e-5
    for P, window in ((37, 8), (1, 128), (5000, 8)):  # 5000 prompts: more than the rank table takes
        hist_d = torch.zeros(P, window, device="cuda")
        seen_d = torch.zeros(P, dtype=torch.int64, device="cuda")
        hist_o, seen_o = np.zeros((P, window)), np.zeros(P, np.int64)
        for batch in range(2):
            pid = rng.integers(0, P, size=wl.B).astype(np.int32)
            R = (wl.rewards + batch).astype(np.float32)
            adv = _misaligned(torch.full((wl.N,), float("nan"), device="cuda"))
            sao.sao_running_mean_advantages(cuda(R), cuda(pid), hist_d, seen_d, m_d, cu_d, adv,
                                            sao.workspace(wl.N))
            torch.cuda.synchronize()
            want, hist_o, seen_o = O.running_mean_advantages(R, pid, wl.loss_mask, wl.cu_seqlens, hist_o, seen_o,
                                                             window)
            assert rel_err_floor(adv.cpu().numpy(), want, 1e-3).max() <= 1e-5
            assert np.array_equal(seen_d.cpu().numpy(), seen_o)
            assert np.allclose(hist_d.cpu().numpy(), hist_o)


# ---------------------------------------------------------------------------
# decoupled three-policy objective (§3.1)
# ---------------------------------------------------------------------------

def _three_policy_inputs(wl, seed):
    """pi_theta = the synthetic log-probs, pi_old = the stale ones, pi_rollout =
    pi_old with an engine mismatch of N(0, 0.3) in log space."""
    rng = np.random.default_rng(seed)
    prox = wl.old_logp_syn.astype(np.float32)
    roll = (prox + rng.normal(0, 0.3, wl.N)).astype(np.float32)
    adv = rng.normal(size=wl.N).astype(np.float32)
    return wl.logp_syn.astype(np.float32), prox, roll, adv


def _decoupled_gpu(logp, prox, roll, adv, mask, el, eh, wl_, wh, n_norm=0):
    N = len(logp)
    loss = torch.empty(1, device="cuda")
    counts = torch.empty(6, dtype=torch.int64, device="cuda")
    coef = torch.full((N,), float("nan"), device="cuda")
    flags = torch.full((N,), 9, dtype=torch.uint8, device="cuda")
    grad = torch.full((N,), float("nan"), device="cuda")
    ws = sao.workspace(N)
    args = [cuda(x) for x in (logp, prox, roll, adv, mask)]
    sao.sao_decoupled_loss_fwd(*args, el, eh, wl_, wh, loss, counts, ws, coef=coef, flags=flags, n_norm=n_norm)
    sao.sao_decoupled_loss_bwd(*args, el, eh, wl_, wh, torch.tensor([0.5], device="cuda"), grad, ws, n_norm=n_norm)
    torch.cuda.synchronize()
    return float(loss.item()), counts.cpu().numpy(), coef.cpu().numpy(), flags.cpu().numpy(), grad.cpu().numpy()


def _near_decoupled_bound(logp, prox, roll, el, eh, wl_, wh, tol=1e-6):
    f64 = lambda x: np.asarray(x, np.float64)
    with np.errstate(all="ignore"):
        r = np.exp(f64(logp) - f64(prox))
        w = np.exp(f64(prox) - f64(roll))
        return ((np.abs(r - (1 - el)) <= tol) | (np.abs(r - (1 + eh)) <= tol) | (np.abs(w - wl_) <= tol) |
                (np.abs(w - wh) <= tol))


def _check_decoupled(logp, prox, roll, adv, mask, el, eh, wl_, wh, n_norm=0):
    loss, counts, coef, flags, grad = _decoupled_gpu(logp, prox, roll, adv, mask, el, eh, wl_, wh, n_norm)
    want = O.decoupled_loss(logp, prox, roll, adv, mask, el, eh, wl_, wh, n_norm)
    skip = _near_decoupled_bound(logp, prox, roll, el, eh, wl_, wh)
    keep = ~skip
    assert np.array_equal(flags[keep], want["flags"][keep])
    if not skip.any():
        assert np.array_equal(counts, want["counts"])
    assert abs(loss - want["loss"]) <= 1e-4 * max(abs(want["loss"]), 1e-6)
    assert rel_err_floor(coef[keep], want["coef"][keep], 1e-12).max() <= 1e-5
    assert rel_err_floor(grad[keep], 0.5 * want["coef"][keep], 1e-12).max() <= 1e-5
    return want


@pytest.mark.parametrize("name", S.CONFIG_NAMES)
def test_decoupled_loss_match_oracle(name):
    wl = S.make_workload(name, dense=False)
    logp, prox, roll, adv = _three_policy_inputs(wl, 11)
    want = _check_decoupled(logp, prox, roll, adv, wl.loss_mask, 0.2, 0.28, 0.5, 2.0)
    assert want["counts"][4] + want["counts"][5] > 0      # the band masks some tokens


def test_decoupled_loss_edge_layouts():
    """Ragged length (not a multiple of 4), non-finite log-probs and advantages,
    masked tokens, an external normaliser and an open upper band."""
    rng = np.random.default_rng(12)
    N = 4099
    logp = (-rng.exponential(2.0, N)).astype(np.float32)
    prox = (logp + rng.normal(0, 0.4, N)).astype(np.float32)
    roll = (prox + rng.normal(0, 0.6, N)).astype(np.float32)
    adv = rng.normal(size=N).astype(np.float32)
    mask = (rng.random(N) < 0.7).astype(np.uint8)
    roll[::97] = -np.inf
    prox[5::101] = np.nan
    adv[7::89] = np.inf
    _check_decoupled(logp, prox, roll, adv, mask, 0.3, 5.0, 0.25, 4.0)
    _check_decoupled(logp, prox, roll, adv, mask, 0.3, 5.0, 0.0, float("inf"), n_norm=1000)
    _check_decoupled(logp[:3], prox[:3], roll[:3], adv[:3], mask[:3], 0.2, 0.28, 0.5, 2.0)


def test_decoupled_loss_equal_old_and_rollout_matches_clip_loss_kernel():
    """pi_old = pi_rollout: the decoupled kernel and the clipped-surrogate
    kernel agree token by token (two independent kernels)."""
    wl = S.make_workload("moe", dense=False)
    logp, prox, _, adv = _three_policy_inputs(wl, 13)
    d = _decoupled_gpu(logp, prox, prox, adv, wl.loss_mask, 0.2, 0.28, 0.5, 2.0)
    c = _clip_gpu(logp, prox, adv, wl.loss_mask, wl.cu_seqlens, 0.2, 0.28, sao.SAO_NORM_TOKEN)
    assert np.array_equal(d[3], c[3]) and np.array_equal(d[1][:4], c[1])
    assert abs(d[0] - c[0]) <= 1e-5 * max(abs(c[0]), 1e-6)
    assert rel_err_floor(d[2], c[2], 1e-12).max() <= 1e-6
