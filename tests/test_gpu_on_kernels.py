"""GPU parity of the O(N) kernels (policy loss, advantages, value loss) with the
fp64 oracle, through the C ABI, on every workload configuration and on edge
cases (empty and ragged inputs, empty trajectories, trajectories without action
tokens, non-finite inputs, misaligned pointers)."""
import numpy as np
import pytest
import torch

from oracle import sao_oracle as O
from paper_2607_07508_gb300 import sao, synthetic as S
from tests._util import cuda, near_bound, rel_err_floor

pytestmark = pytest.mark.gpu

ADV_TOL = 1e-5      # relative to max(|A|, 1e-3)
LOSS_TOL = 1e-4     # relative


def f32(x):
    """The ABI takes fp32 scalars; the oracle gets the same rounded values."""
    return float(np.float32(x))


def _gae_gpu(wl, values=None, mask=None, gamma=None, lam=None, lam_c=None, alpha=None):
    values = wl.values if values is None else values
    mask = wl.loss_mask if mask is None else mask
    N = len(values)
    g = dict(gamma=wl.gamma if gamma is None else gamma, lam=wl.lam if lam is None else lam,
             lam_c=wl.lam_critic if lam_c is None else lam_c, alpha=wl.alpha if alpha is None else alpha)
    g = {k: f32(x) for k, x in g.items()}
    adv = torch.empty(N, dtype=torch.float32, device="cuda")
    ret = torch.empty(N, dtype=torch.float32, device="cuda")
    ws = sao.workspace(N)
    sao.sao_advantages(cuda(values), cuda(wl.rewards), cuda(mask), cuda(wl.cu_seqlens), g["gamma"], g["lam"],
                       g["lam_c"], g["alpha"], adv, ret, ws)
    torch.cuda.synchronize()
    return adv.cpu().numpy(), ret.cpu().numpy(), g


@pytest.mark.parametrize("name", S.CONFIG_NAMES)
def test_advantages_match_oracle(name):
    wl = S.make_workload(name, dense=False)
    adv, ret, g = _gae_gpu(wl)
    want_a, want_r = O.advantages(wl.values, wl.rewards, wl.loss_mask, wl.cu_seqlens, g["gamma"], g["lam"],
                                  g["lam_c"], g["alpha"])
    assert rel_err_floor(adv, want_a, 1e-3).max() <= ADV_TOL
    assert rel_err_floor(ret, want_r, 1e-3).max() <= ADV_TOL


@pytest.mark.parametrize("gamma,lam,lam_c,alpha", [(1.0, 0.95, 1.0, 0.0), (0.99, 0.9, 0.97, 0.0),
                                                   (1.0, 1.0, 1.0, 1.5), (0.97, 1.0, 1.0, 1.5),
                                                   (0.5, 0.0, 0.3, 0.0)])
def test_advantages_coefficients(gamma, lam, lam_c, alpha):
    wl = S.make_workload("moe", dense=False)
    adv, ret, g = _gae_gpu(wl, gamma=gamma, lam=lam, lam_c=lam_c, alpha=alpha)
    want_a, want_r = O.advantages(wl.values, wl.rewards, wl.loss_mask, wl.cu_seqlens, g["gamma"], g["lam"],
                                  g["lam_c"], g["alpha"])
    assert rel_err_floor(adv, want_a, 1e-3).max() <= ADV_TOL
    assert rel_err_floor(ret, want_r, 1e-3).max() <= ADV_TOL


@pytest.mark.parametrize("lengths", [[1], [5, 0, 0, 7], [0, 4096, 1, 4095, 0], [4097, 13, 8190],
                                     [3] * 2000, [70001], [0, 0, 17, 0]])
def test_advantages_edge_layouts(lengths):
    wl = S.make_custom(lengths, 8, 16, "f32", seed=sum(lengths) + len(lengths), dense=False, obs_frac=0.4)
    wl.loss_mask[::97] = 0
    adv, ret, g = _gae_gpu(wl, gamma=0.99, lam=0.95, lam_c=1.0, alpha=1.5)
    want_a, want_r = O.advantages(wl.values, wl.rewards, wl.loss_mask, wl.cu_seqlens, g["gamma"], g["lam"],
                                  g["lam_c"], g["alpha"])
    assert rel_err_floor(adv, want_a, 1e-3).max() <= ADV_TOL
    assert rel_err_floor(ret, want_r, 1e-3).max() <= ADV_TOL


@pytest.mark.parametrize("lengths", [[1], [5, 0, 0, 7], [0, 4096, 1, 4095, 0], [4097, 13, 8190],
                                     [3] * 2000, [70001], [0, 0, 17, 0]])
@pytest.mark.parametrize("offset", [0, 1])
def test_advantages_telescoped_edge_layouts(lengths, offset):
    """gamma = lambda = lambda_critic = 1 (no length-adaptive lambda) takes the
    one-pass telescoped kernel: ragged layouts, empty trajectories and
    trajectories without action tokens, with 16-byte aligned and misaligned
    (one element off) inputs and outputs."""
    wl = S.make_custom(lengths, 8, 16, "f32", seed=sum(lengths) + 7 * len(lengths), dense=False, obs_frac=0.4)
    wl.loss_mask[::97] = 0
    N = wl.N

    def shifted(a, dtype):
        t = torch.zeros(N + offset, dtype=dtype, device="cuda")
        t[offset:] = torch.as_tensor(a).to(dtype).cuda()
        return t[offset:]

    v, m = shifted(wl.values, torch.float32), shifted(wl.loss_mask, torch.uint8)
    adv = torch.full((N + offset,), float("nan"), device="cuda")[offset:]
    ret = torch.full((N + offset,), float("nan"), device="cuda")[offset:]
    sao.sao_advantages(v, cuda(wl.rewards), m, cuda(wl.cu_seqlens), 1.0, 1.0, 1.0, 0.0, adv, ret, sao.workspace(N))
    torch.cuda.synchronize()
    want_a, want_r = O.advantages(wl.values, wl.rewards, wl.loss_mask, wl.cu_seqlens, 1.0, 1.0, 1.0, 0.0)
    assert rel_err_floor(adv.cpu().numpy(), want_a, 1e-3).max() <= ADV_TOL
    assert rel_err_floor(ret.cpu().numpy(), want_r, 1e-3).max() <= ADV_TOL


@pytest.mark.parametrize("lengths", [[1], [5, 0, 0, 7], [0, 4096, 1, 4095, 0], [4097, 13, 8190],
                                     [3] * 2000, [70001], [0, 0, 17, 0], [0] * 3 + [300000, 0, 77777, 1] + [0] * 2])
@pytest.mark.parametrize("offset", [0, 1])
@pytest.mark.parametrize("gamma,lam,lam_c", [(1.0, 0.95, 1.0), (0.99, 0.9, 0.97)])
def test_advantages_fixed_lambda_layouts(lengths, offset, gamma, lam, lam_c):
    """A fixed lambda (alpha = 0) takes the one-launch set-up (a thread per
    trajectory writes the chunk_first entries of the sub-chunks starting
    inside it, so empty trajectories write none) and the scan; aligned inputs
    take the tensor copies for whole chunks and plain loads for the ragged
    end, inputs and outputs one element off 16-byte alignment take plain loads
    and stores everywhere."""
    wl = S.make_custom(lengths, 8, 16, "f32", seed=sum(lengths) + 11 * len(lengths), dense=False, obs_frac=0.4)
    wl.loss_mask[::97] = 0
    N = wl.N

    def shifted(a, dtype):
        t = torch.zeros(N + offset, dtype=dtype, device="cuda")
        t[offset:] = torch.as_tensor(a).to(dtype).cuda()
        return t[offset:]

    v, m = shifted(wl.values, torch.float32), shifted(wl.loss_mask, torch.uint8)
    adv = torch.full((N + offset,), float("nan"), device="cuda")[offset:]
    ret = torch.full((N + offset,), float("nan"), device="cuda")[offset:]
    g, l, lc = f32(gamma), f32(lam), f32(lam_c)
    sao.sao_advantages(v, cuda(wl.rewards), m, cuda(wl.cu_seqlens), g, l, lc, 0.0, adv, ret, sao.workspace(N))
    torch.cuda.synchronize()
    want_a, want_r = O.advantages(wl.values, wl.rewards, wl.loss_mask, wl.cu_seqlens, g, l, lc, 0.0)
    assert rel_err_floor(adv.cpu().numpy(), want_a, 1e-3).max() <= ADV_TOL
    assert rel_err_floor(ret.cpu().numpy(), want_r, 1e-3).max() <= ADV_TOL


def test_advantages_no_action_tokens_and_empty():
    wl = S.make_custom([10, 0, 300], 8, 16, "f32", seed=3, dense=False)
    wl.loss_mask[:] = 0
    adv, ret, _ = _gae_gpu(wl)
    assert np.all(adv == 0) and np.all(ret == 0)


def test_advantages_bandwidth_size_properties():
    """2^27 tokens: gamma = lambda = 1 gives A = R - V exactly on action tokens
    and ret = R (telescoping), and sampled trajectories match the oracle."""
    wl = S.bandwidth_workload()
    adv, ret, _ = _gae_gpu(wl, gamma=1.0, lam=1.0, lam_c=1.0, alpha=0.0)
    m = wl.loss_mask.astype(bool)
    traj = np.repeat(np.arange(wl.B), np.diff(wl.cu_seqlens))
    R = wl.rewards[traj]
    want = R.astype(np.float64) - wl.values
    assert rel_err_floor(adv[m], want[m], 1e-3).max() <= ADV_TOL
    assert np.all(ret[m] == R[m]) and np.all(adv[~m] == 0) and np.all(ret[~m] == 0)
    adv, ret, _ = _gae_gpu(wl, gamma=1.0, lam=0.95, lam_c=1.0, alpha=1.5)
    rng = np.random.default_rng(0)
    for b in rng.choice(wl.B, size=24, replace=False):
        lo, hi = wl.cu_seqlens[b], wl.cu_seqlens[b + 1]
        a, r = O.advantages(wl.values[lo:hi], wl.rewards[b:b + 1], wl.loss_mask[lo:hi], np.array([0, hi - lo]),
                            1.0, f32(0.95), 1.0, 1.5)
        assert rel_err_floor(adv[lo:hi], a, 1e-3).max() <= ADV_TOL
        assert rel_err_floor(ret[lo:hi], r, 1e-3).max() <= ADV_TOL


@pytest.mark.parametrize("N", [(1 << 23) + 4321, (1 << 24) + 77, 1 << 25, (1 << 26) + 12345])
def test_advantages_long_lane_segments(N):
    """From 2^23 tokens on, the scan's lanes own 64-token segments (two chunks
    in flight per warp), from 2^25 on 128-token segments (one chunk at a
    time), streamed in 32-token pieces: 64 sampled trajectories and the last
    two (the ragged tail) against the oracle, with lambda = 0.95 and with the
    length-adaptive lambda and lambda_critic < 1."""
    wl = S.bandwidth_workload(N=N, B=max(1, N >> 13))
    rng = np.random.default_rng(N % 1000)
    picks = np.concatenate([rng.choice(wl.B, size=64, replace=False), [wl.B - 2, wl.B - 1]])
    for coefs in ((1.0, 0.95, 1.0, 0.0), (0.99, 1.0, 0.97, 1.5)):
        adv, ret, g = _gae_gpu(wl, gamma=coefs[0], lam=coefs[1], lam_c=coefs[2], alpha=coefs[3])
        for b in picks:
            lo, hi = wl.cu_seqlens[b], wl.cu_seqlens[b + 1]
            a, r = O.advantages(wl.values[lo:hi], wl.rewards[b:b + 1], wl.loss_mask[lo:hi], np.array([0, hi - lo]),
                                g["gamma"], g["lam"], g["lam_c"], g["alpha"])
            assert rel_err_floor(adv[lo:hi], a, 1e-3).max() <= ADV_TOL
            assert rel_err_floor(ret[lo:hi], r, 1e-3).max() <= ADV_TOL


def test_advantages_misaligned_4_piece_mode():
    """2^26 + 999 tokens (4-piece lane segments, one chunk per warp) with
    values, mask and outputs one element off 16-byte alignment: no tensor
    maps, every piece staged with plain loads and stored with plain stores;
    sampled trajectories and the ragged tail against the oracle."""
    N = (1 << 26) + 999
    wl = S.bandwidth_workload(N=N, B=N >> 13)
    off = 1

    def shifted(a, dtype):
        t = torch.zeros(N + off, dtype=dtype, device="cuda")
        t[off:] = torch.as_tensor(a).to(dtype).cuda()
        return t[off:]

    v, m = shifted(wl.values, torch.float32), shifted(wl.loss_mask, torch.uint8)
    adv = torch.full((N + off,), float("nan"), device="cuda")[off:]
    ret = torch.full((N + off,), float("nan"), device="cuda")[off:]
    g, l = f32(1.0), f32(0.95)
    sao.sao_advantages(v, cuda(wl.rewards), m, cuda(wl.cu_seqlens), g, l, 1.0, 0.0, adv, ret, sao.workspace(N))
    torch.cuda.synchronize()
    adv, ret = adv.cpu().numpy(), ret.cpu().numpy()
    rng = np.random.default_rng(7)
    picks = np.concatenate([rng.choice(wl.B, size=32, replace=False), [wl.B - 2, wl.B - 1]])
    for b in picks:
        lo, hi = wl.cu_seqlens[b], wl.cu_seqlens[b + 1]
        a, r = O.advantages(wl.values[lo:hi], wl.rewards[b:b + 1], wl.loss_mask[lo:hi], np.array([0, hi - lo]),
                            g, l, 1.0, 0.0)
        assert rel_err_floor(adv[lo:hi], a, 1e-3).max() <= ADV_TOL
        assert rel_err_floor(ret[lo:hi], r, 1e-3).max() <= ADV_TOL


def test_advantages_short_trajectories_random_masks():
    """4-piece lane segments (2^25 tokens and more, one chunk per warp in all
    of its TMEM columns) with ~512-token trajectories and token-by-token random
    masks: many trajectory ends inside each piece (the per-token path) and
    mixed 4-token groups; sampled trajectories and the ragged tail against the
    oracle."""
    N = (1 << 26) + 999
    wl = S.bandwidth_workload(N=N, B=N >> 9)
    rng = np.random.default_rng(26)
    wl.loss_mask = (rng.random(N) < 0.6).astype(np.uint8)
    picks = np.concatenate([rng.choice(wl.B, size=64, replace=False), [wl.B - 2, wl.B - 1]])
    for coefs in ((1.0, 0.95, 1.0, 0.0), (0.99, 1.0, 0.97, 1.5)):
        adv, ret, g = _gae_gpu(wl, gamma=coefs[0], lam=coefs[1], lam_c=coefs[2], alpha=coefs[3])
        for b in picks:
            lo, hi = wl.cu_seqlens[b], wl.cu_seqlens[b + 1]
            a, r = O.advantages(wl.values[lo:hi], wl.rewards[b:b + 1], wl.loss_mask[lo:hi], np.array([0, hi - lo]),
                                g["gamma"], g["lam"], g["lam_c"], g["alpha"])
            assert rel_err_floor(adv[lo:hi], a, 1e-3).max() <= ADV_TOL
            assert rel_err_floor(ret[lo:hi], r, 1e-3).max() <= ADV_TOL


def test_advantages_checked_mode_reports_bad_cu_seqlens():
    wl = S.make_custom([10, 20], 8, 16, "f32", seed=5, dense=False)
    bad = wl.cu_seqlens.copy()
    bad[1] = 25
    bad[2] = 15          # decreasing
    ws = sao.workspace(30)
    adv = torch.empty(30, device="cuda")
    ret = torch.empty(30, device="cuda")
    sao.sao_set_checked(True)
    try:
        with pytest.raises(sao.SaoError) as e:
            sao.sao_advantages(cuda(wl.values), cuda(wl.rewards), cuda(wl.loss_mask), cuda(bad), 1.0, 1.0, 1.0,
                               0.0, adv, ret, ws)
        assert e.value.status == 6
        sao.sao_advantages(cuda(wl.values), cuda(wl.rewards), cuda(wl.loss_mask), cuda(wl.cu_seqlens), 1.0, 1.0,
                           1.0, 0.0, adv, ret, ws)
    finally:
        sao.sao_set_checked(False)


# ---------------------------------------------------------------------------
# policy loss
# ---------------------------------------------------------------------------

def _pl_gpu(logp, old, adv, mask, el, eh, n_norm=0, offset=0):
    N = len(logp)
    pad = lambda a: np.concatenate([np.zeros(offset, a.dtype), a]) if offset else a
    tl, to, ta, tm = (cuda(pad(x)) for x in (logp, old, adv, mask))
    sl = lambda t: t[offset:] if offset else t
    loss = torch.empty(1, device="cuda")
    counts = torch.empty(4, dtype=torch.int64, device="cuda")
    coef = torch.empty(N + offset, device="cuda")
    flags = torch.empty(N + offset, dtype=torch.uint8, device="cuda")
    ws = sao.workspace(N)
    sao.sao_policy_loss_fwd(sl(tl), sl(to), sl(ta), sl(tm), el, eh, loss, counts, ws, coef=sl(coef),
                            flags=sl(flags), n_norm=n_norm)
    gl = torch.tensor([0.75], device="cuda")
    grad = torch.empty(N + offset, device="cuda")
    sao.sao_policy_loss_bwd(sl(tl), sl(to), sl(ta), sl(tm), el, eh, gl, sl(grad), ws, n_norm=n_norm)
    torch.cuda.synchronize()
    return (float(loss.item()), counts.cpu().numpy(), sl(coef).cpu().numpy(), sl(flags).cpu().numpy(),
            sl(grad).cpu().numpy())


def _check_pl(logp, old, adv, mask, el, eh, n_norm=0, offset=0):
    loss, counts, coef, flags, grad = _pl_gpu(logp, old, adv, mask, el, eh, n_norm, offset)
    want = O.policy_loss(logp, old, adv, mask, el, eh, n_norm)
    skip = near_bound(logp, old, el, eh) & (mask == 1)
    assert np.array_equal(flags[~skip], want["flags"][~skip])
    if not skip.any():
        assert np.array_equal(counts, want["counts"])
    else:
        assert counts[0] == want["counts"][0]
        assert abs(int(counts[1:3].sum()) - int(want["counts"][1:3].sum())) <= int(skip.sum())
    wl = want["loss"]
    assert abs(loss - wl) <= LOSS_TOL * max(abs(wl), 1e-6)
    keep = ~skip
    assert rel_err_floor(coef[keep], want["coef"][keep], 1e-12).max() <= 1e-5
    assert rel_err_floor(grad[keep], 0.75 * want["coef"][keep], 1e-12).max() <= 1e-5
    return want


@pytest.mark.parametrize("name", S.CONFIG_NAMES)
def test_policy_loss_match_oracle(name):
    wl = S.make_workload(name, dense=False)
    adv, _ = O.advantages(wl.values, wl.rewards, wl.loss_mask, wl.cu_seqlens, wl.gamma, wl.lam, wl.lam_critic,
                          wl.alpha)
    adv = adv.astype(np.float32)
    want = _check_pl(wl.logp_syn, wl.old_logp_syn, adv, wl.loss_mask, wl.eps_low, wl.eps_high)
    if name == "large":
        assert want["counts"][1] > 0 and want["counts"][2] > 0


def test_policy_loss_edge_cases():
    rng = np.random.default_rng(7)
    for N in (1, 3, 4, 5, 1023, 4097):
        logp = (-rng.exponential(2.0, N)).astype(np.float32)
        old = (logp + rng.normal(0, 0.3, N)).astype(np.float32)
        adv = rng.normal(size=N).astype(np.float32)
        mask = (rng.random(N) < 0.7).astype(np.uint8)
        _check_pl(logp, old, adv, mask, 0.2, 0.28)
        _check_pl(logp, old, adv, mask, 0.3, 5.0, n_norm=12345)
        _check_pl(logp, old, adv, mask, 0.8, 3.0, offset=1)     # misaligned: scalar path
        _check_pl(logp, old, adv, mask, 0.8, 3.0, n_norm=777, offset=1)  # forward counts the action tokens
    # non-finite inputs, masked tokens, exact-bound ratios, eps_low >= 1
    logp = np.array([-1, -1, -1, -1, -1, -30, -1, -1], np.float32)
    old = np.array([-np.inf, -1, np.nan, -1, -1, 0, -1.5, -1], np.float32)
    adv = np.array([1, np.nan, 1, 1, np.inf, 1, 1, 2], np.float32)
    mask = np.array([1, 1, 1, 0, 1, 1, 1, 1], np.uint8)
    _check_pl(logp, old, adv, mask, 1.0, 0.28)
    _check_pl(logp, old, adv, mask, 0.2, 0.28)


def test_policy_loss_empty():
    loss, counts, _, _, _ = _pl_gpu(np.zeros(0, np.float32), np.zeros(0, np.float32), np.zeros(0, np.float32),
                                    np.zeros(0, np.uint8), 0.2, 0.28)
    assert loss == 0.0 and list(counts) == [0, 0, 0, 0]


def test_policy_loss_bandwidth_size():
    wl = S.bandwidth_workload()
    adv = (np.random.default_rng(1).standard_normal(wl.N, dtype=np.float32))
    _check_pl(wl.logp_syn, wl.old_logp_syn, adv, wl.loss_mask, wl.eps_low, wl.eps_high)
    # with the normaliser given, the forward counts the action tokens itself
    _check_pl(wl.logp_syn, wl.old_logp_syn, adv, wl.loss_mask, wl.eps_low, wl.eps_high, n_norm=int(wl.N))


# ---------------------------------------------------------------------------
# value loss
# ---------------------------------------------------------------------------

def _vl_gpu(v, r, m, n_norm=0):
    N = len(v)
    loss = torch.empty(1, device="cuda")
    grad = torch.empty(N, device="cuda")
    ev = torch.empty(4, dtype=torch.float64, device="cuda")
    sao.sao_value_loss(cuda(v), cuda(r), cuda(m), loss, grad, sao.workspace(N), ev_sums=ev, n_norm=n_norm)
    torch.cuda.synchronize()
    return float(loss.item()), grad.cpu().numpy(), ev.cpu().numpy()


@pytest.mark.parametrize("name", S.CONFIG_NAMES + ("bandwidth",))
def test_value_loss_match_oracle(name):
    wl = S.bandwidth_workload() if name == "bandwidth" else S.make_workload(name, dense=False)
    rng = np.random.default_rng(2)
    ret = (wl.values + rng.normal(0, 0.3, wl.N)).astype(np.float32)
    for n_norm in (0, 3 * int(wl.loss_mask.sum()) + 1):  # counted, or given (one pass)
        loss, grad, ev = _vl_gpu(wl.values, ret, wl.loss_mask, n_norm)
        wl_, wg, wev = O.value_loss(wl.values, ret, wl.loss_mask, n_norm)
        assert abs(loss - wl_) <= LOSS_TOL * abs(wl_)
        assert rel_err_floor(grad, wg, 1e-12).max() <= 1e-5
        # exact per-token terms (two-sum, fused-multiply-add remainders), compensated
        # fp32 sums per thread, fp64 across threads: fp64-grade sums
        assert np.allclose(ev, wev, rtol=1e-9, atol=1e-9 * np.abs(wev).max())


def test_value_loss_zero_and_empty():
    v = np.random.default_rng(3).normal(size=1001).astype(np.float32)
    m = np.ones(1001, np.uint8)
    loss, grad, ev = _vl_gpu(v, v, m)
    assert loss == 0.0 and np.all(grad == 0.0)
    loss, grad, ev = _vl_gpu(v, v + 1, np.zeros(1001, np.uint8))
    assert loss == 0.0 and np.all(grad == 0.0) and np.all(ev == 0.0)
