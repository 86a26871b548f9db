"""GPU parity of the tensor-core GEMMs tiled over CTA pairs (clusters of 2,
tcgen05.mma.cta_group::2 with M = 256; sao_set_cta_pairs(1)) with the fp64
oracle and with the single-CTA tiling, through the C ABI: ragged shapes with
every tile of the pair partly out of range, the cached path, two M tiles per
pair tile, vocabulary chunks and row blocks, and the moe shape. Checked mode
is on, so a pipeline wait that gives up fails the call instead of passing
garbage."""
import numpy as np
import pytest
import torch

from oracle import sao_oracle as O
from paper_2607_07508_gb300 import sao, synthetic as S
from tests._util import rel_l2
from tests.test_gpu_logprobs_full import oracle_dW_sample

pytestmark = pytest.mark.gpu

LOGP_TOL = 2e-3     # absolute
GRAD_TOL = 2e-2     # relative L2
DEFAULT_DZ_BUDGET = 4 << 30


@pytest.fixture(autouse=True)
def pairs_checked():
    sao.sao_set_cta_pairs(True)
    sao.sao_set_checked(1)
    try:
        yield
    finally:
        sao.sao_set_checked(0)
        sao.sao_set_cta_pairs(False)


def _case(N, h, V, seed):
    wl = S.make_custom([N], h, V, "bf16", seed=seed, device="cuda")
    return wl, wl.H, wl.W, torch.as_tensor(wl.y).cuda()


def _fwd_bwd(H, W, y, G, row_mask=None, cache=None):
    N, h = H.shape
    V = W.shape[0]
    ws = sao.workspace(N, h, V, H.dtype)
    logp = torch.empty(N, device="cuda")
    lse = torch.empty(N, device="cuda")
    dH = torch.full_like(H, float("nan"))
    dW = torch.full((V, h), float("nan"), device="cuda")
    if cache is None:
        sao.sao_token_logprobs_fwd(H, W, y, logp, lse, ws, row_mask=row_mask)
        sao.sao_token_logprobs_bwd(H, W, y, lse, G, dH, dW, ws)
    else:
        sao.sao_token_logprobs_fwd_cached(H, W, y, logp, lse, cache, ws, row_mask=row_mask)
        sao.sao_token_logprobs_bwd_cached(H, W, y, lse, G, dH, dW, cache, ws)
    torch.cuda.synchronize()
    return logp, lse, dH, dW


def _single_cta(fn):
    sao.sao_set_cta_pairs(False)
    try:
        return fn()
    finally:
        sao.sao_set_cta_pairs(True)


CASES = [(1, 8, 1), (129, 64, 257), (300, 192, 1000), (513, 520, 2000), (1000, 256, 4113), (2048, 256, 20000)]


@pytest.mark.parametrize("N,h,V", CASES)
def test_pairs_match_oracle_and_single_cta(N, h, V):
    assert sao.sao_get_cta_pairs()
    wl, H, W, y = _case(N, h, V, seed=3 * N + h + V)
    rng = np.random.default_rng(N + 1)
    G = rng.normal(size=N).astype(np.float32)
    G[rng.random(N) < 0.3] = 0.0
    Gt = torch.as_tensor(G).cuda()
    logp, lse, dH, dW = _fwd_bwd(H, W, y, Gt)
    want_lp, want_lse = O.token_logprobs(H.cpu(), W.cpu(), wl.y)
    assert np.abs(logp.cpu().numpy() - want_lp).max() <= LOGP_TOL
    assert np.abs(lse.cpu().numpy() - want_lse).max() <= LOGP_TOL
    want_dH, want_dW = O.token_logprobs_bwd(H.cpu(), W.cpu(), wl.y, want_lse, G)
    got_dH = dH.float().cpu().numpy()
    assert rel_l2(got_dH, want_dH) <= GRAD_TOL
    assert rel_l2(dW.cpu().numpy(), want_dW) <= GRAD_TOL
    assert np.all(got_dH[G == 0] == 0)
    # the single-CTA tiling: the same sums in the same K order per output element
    lp1, lse1, dH1, dW1 = _single_cta(lambda: _fwd_bwd(H, W, y, Gt))
    assert torch.allclose(logp, lp1, atol=1e-5, rtol=0)
    assert rel_l2(dH.float().cpu().numpy(), dH1.float().cpu().numpy()) <= 1e-3
    assert rel_l2(dW.cpu().numpy(), dW1.cpu().numpy()) <= 1e-3


@pytest.mark.parametrize("N,h,V", [(300, 192, 1000), (2048, 256, 20000)])
def test_pairs_cached_path(N, h, V):
    wl, H, W, y = _case(N, h, V, seed=5 * N + V)
    rng = np.random.default_rng(N + 2)
    G = rng.normal(size=N).astype(np.float32)
    G[rng.random(N) < 0.3] = 0.0
    mask = torch.as_tensor(wl.loss_mask).cuda()
    G[wl.loss_mask == 0] = 0.0
    cache = sao.logprob_cache(N, V)
    logp, lse, dH, dW = _fwd_bwd(H, W, y, torch.as_tensor(G).cuda(), row_mask=mask, cache=cache)
    m = wl.loss_mask.astype(bool)
    want_lp, want_lse = O.token_logprobs(H.cpu(), W.cpu(), wl.y)
    assert np.abs(logp.cpu().numpy()[m] - want_lp[m]).max() <= LOGP_TOL
    want_dH, want_dW = O.token_logprobs_bwd(H.cpu(), W.cpu(), wl.y, want_lse, G)
    assert rel_l2(dH.float().cpu().numpy(), want_dH) <= GRAD_TOL
    assert rel_l2(dW.cpu().numpy(), want_dW) <= GRAD_TOL


def test_pairs_chunks_and_row_blocks():
    """A 1 MiB dZ bound: many row blocks and vocabulary chunks, each GEMM with
    ragged pair tiles; dW accumulates across the blocks."""
    wl, H, W, y = _case(3000, 256, 5000, seed=17)
    G = np.random.default_rng(4).normal(size=3000).astype(np.float32)
    sao.sao_set_dz_budget_bytes(1 << 20)
    try:
        logp, lse, dH, dW = _fwd_bwd(H, W, y, torch.as_tensor(G).cuda())
    finally:
        sao.sao_set_dz_budget_bytes(DEFAULT_DZ_BUDGET)
    _, want_lse = O.token_logprobs(H.cpu(), W.cpu(), wl.y)
    want_dH, want_dW = O.token_logprobs_bwd(H.cpu(), W.cpu(), wl.y, want_lse, G)
    assert rel_l2(dH.float().cpu().numpy(), want_dH) <= GRAD_TOL
    assert rel_l2(dW.cpu().numpy(), want_dW) <= GRAD_TOL


def test_pairs_two_m_tiles_per_pair_tile():
    """20,100 rows x 20,168 vocabulary rows at h = 2048: both backward GEMMs take
    two 256-row M tiles per pair tile (enough tiles for four waves of pairs);
    sampled rows against the oracle, everything against the single-CTA run."""
    N, h, V = 20100, 2048, 20168
    wl, H, W, y = _case(N, h, V, seed=23)
    rng = np.random.default_rng(6)
    G = (rng.normal(size=N) * 1e-2).astype(np.float32)
    Gt = torch.as_tensor(G).cuda()
    logp, lse, dH, dW = _fwd_bwd(H, W, y, Gt)
    rows = np.sort(rng.choice(N, size=256, replace=False))
    Hs = H[torch.as_tensor(rows).cuda()].cpu()
    want_lp, want_lse = O.token_logprobs(Hs, W.cpu(), wl.y[rows])
    assert np.abs(logp.cpu().numpy()[rows] - want_lp).max() <= LOGP_TOL
    want_dH, _ = O.token_logprobs_bwd(Hs, W.cpu(), wl.y[rows], want_lse, G[rows])
    assert rel_l2(dH[torch.as_tensor(rows).cuda()].float().cpu().numpy(), want_dH) <= GRAD_TOL
    vrows = np.unique(np.concatenate([rng.choice(V, size=128, replace=False), wl.y[rows[:16]], [V - 1]]))
    want_dW = oracle_dW_sample(H, W.cpu(), wl.y, lse.cpu().numpy().astype(np.float64), G.astype(np.float64), vrows)
    assert rel_l2(dW[torch.as_tensor(vrows).cuda()].cpu().numpy(), want_dW) <= GRAD_TOL
    lp1, _, dH1, dW1 = _single_cta(lambda: _fwd_bwd(H, W, y, Gt))
    assert torch.allclose(logp, lp1, atol=1e-5, rtol=0)
    assert rel_l2(dH.float().cpu().numpy(), dH1.float().cpu().numpy()) <= 1e-3
    assert rel_l2(dW.cpu().numpy(), dW1.cpu().numpy()) <= 1e-3


def test_pairs_moe_shape_bench_calls():
    """The moe shape as bench.py calls it (forward on the action rows, dense
    gradient on them), with pairs, against the single-CTA run and sampled rows
    against the oracle."""
    wl = S.make_workload("moe", device="cuda")
    N, h, V = wl.N, wl.h, wl.V
    y = torch.as_tensor(wl.y).cuda()
    mask = torch.as_tensor(wl.loss_mask).cuda()
    rng = np.random.default_rng(8)
    G = (rng.normal(size=N) * 1e-4).astype(np.float32)
    G[wl.loss_mask == 0] = 0.0
    Gt = torch.as_tensor(G).cuda()
    logp, lse, dH, dW = _fwd_bwd(wl.H, wl.W, y, Gt, row_mask=mask)
    lp1, _, dH1, dW1 = _single_cta(lambda: _fwd_bwd(wl.H, wl.W, y, Gt, row_mask=mask))
    assert torch.allclose(logp, lp1, atol=1e-5, rtol=0)
    d = (dH.float() - dH1.float()).norm() / dH1.float().norm()
    assert d.item() <= 1e-3
    d = (dW - dW1).norm() / dW1.norm()
    assert d.item() <= 1e-3
    rows = np.sort(rng.choice(np.flatnonzero(wl.loss_mask), size=256, replace=False))
    Hs = wl.H[torch.as_tensor(rows).cuda()].cpu()
    want_lp, want_lse = O.token_logprobs(Hs, wl.W.cpu(), wl.y[rows])
    assert np.abs(logp.cpu().numpy()[rows] - want_lp).max() <= LOGP_TOL
    want_dH, _ = O.token_logprobs_bwd(Hs, wl.W.cpu(), wl.y[rows], want_lse, G[rows])
    assert rel_l2(dH[torch.as_tensor(rows).cuda()].float().cpu().numpy(), want_dH) <= GRAD_TOL
