"""GPU parity of the cached log-prob path (sao_token_logprobs_fwd_cached /
_bwd_cached: the forward stores bf16 e = exp(z - kappa) with one shift per row,
the backward runs its two GEMMs on e with per-row scales instead of recomputing
the logits) with the fp64 oracle, through the C ABI: small shapes with ragged
tiles checked in full, the moe shape in the launch configuration bench.py
times checked on sampled rows, row masks, vocabulary chunking, accumulation,
rows beyond the stored range and the argument errors."""
import numpy as np
import pytest
import torch

from oracle import sao_oracle as O
from paper_2607_07508_gb300 import sao, synthetic as S
from tests._util import rel_l2

pytestmark = pytest.mark.gpu

LOGP_TOL = 2e-3     # absolute
GRAD_TOL = 2e-2     # relative L2
DEFAULT_DZ_BUDGET = 4 << 30   # the library's default bound on the backward's dZ buffer


def _fwd(H, W, y, cache, row_mask=None):
    N, h = H.shape
    V = W.shape[0]
    logp = torch.empty(N, device="cuda")
    lse = torch.empty(N, device="cuda")
    ws = sao.workspace(N, h, V, H.dtype)
    sao.sao_token_logprobs_fwd_cached(H, W, y, logp, lse, cache, ws, row_mask=row_mask)
    return logp, lse


def _bwd(H, W, y, lse, G, cache, accumulate=None):
    N, h = H.shape
    V = W.shape[0]
    dH = torch.full_like(H, float("nan"))
    dW = accumulate.clone() if accumulate is not None else torch.full((V, h), float("nan"), device="cuda")
    ws = sao.workspace(N, h, V, H.dtype)
    sao.sao_token_logprobs_bwd_cached(H, W, y, lse, G, dH, dW, cache, ws, accumulate_dW=accumulate is not None)
    return dH, dW


def _case(N, h, V, seed):
    wl = S.make_custom([N], h, V, "bf16", seed=seed, device="cuda")
    return wl, wl.H, wl.W, torch.as_tensor(wl.y).cuda()


CASES = [(300, 192, 1000), (1000, 256, 4113), (129, 64, 257), (1, 8, 1), (513, 520, 2000), (2048, 256, 20000)]


@pytest.mark.parametrize("N,h,V", CASES)
def test_cached_forward_and_backward_match_oracle(N, h, V):
    wl, H, W, y = _case(N, h, V, seed=N + h + V + 1)
    cache = sao.logprob_cache(N, V)
    logp, lse = _fwd(H, W, y, cache)
    rng = np.random.default_rng(N + 7)
    G = rng.normal(size=N).astype(np.float32)
    G[rng.random(N) < 0.3] = 0.0
    dH, dW = _bwd(H, W, y, lse, torch.as_tensor(G).cuda(), cache)
    torch.cuda.synchronize()
    want_lp, want_lse = O.token_logprobs(H.cpu(), W.cpu(), wl.y)
    assert np.abs(logp.cpu().numpy() - want_lp).max() <= LOGP_TOL
    assert np.abs(lse.cpu().numpy() - want_lse).max() <= LOGP_TOL
    want_dH, want_dW = O.token_logprobs_bwd(H.cpu(), W.cpu(), wl.y, want_lse, G)
    got_dH = dH.float().cpu().numpy()
    assert rel_l2(got_dH, want_dH) <= GRAD_TOL
    assert rel_l2(dW.cpu().numpy(), want_dW) <= GRAD_TOL
    assert np.all(got_dH[G == 0] == 0)


def test_cached_path_agrees_with_recompute_path():
    """Same inputs through both paths: identical log-probs (the forward's
    softmax is the same arithmetic) and gradients within the bf16 rounding of
    the stored probabilities."""
    wl, H, W, y = _case(777, 256, 5000, seed=31)
    cache = sao.logprob_cache(777, 5000)
    lp_c, lse_c = _fwd(H, W, y, cache)
    ws = sao.workspace(777, 256, 5000, H.dtype)
    lp_r = torch.empty(777, device="cuda")
    lse_r = torch.empty(777, device="cuda")
    sao.sao_token_logprobs_fwd(H, W, y, lp_r, lse_r, ws)
    G = torch.as_tensor(np.random.default_rng(8).normal(size=777).astype(np.float32)).cuda()
    dH_c, dW_c = _bwd(H, W, y, lse_c, G, cache)
    dH_r = torch.empty_like(H)
    dW_r = torch.empty(5000, 256, device="cuda")
    sao.sao_token_logprobs_bwd(H, W, y, lse_r, G, dH_r, dW_r, ws)
    torch.cuda.synchronize()
    assert torch.allclose(lse_c, lse_r, atol=1e-5) and torch.allclose(lp_c, lp_r, atol=1e-5)
    assert rel_l2(dH_c.float().cpu().numpy(), dH_r.float().cpu().numpy()) <= 1e-2
    assert rel_l2(dW_c.cpu().numpy(), dW_r.cpu().numpy()) <= 1e-2


def test_cached_row_mask_and_skipped_rows():
    """Forward on masked rows only; a gradient on a skipped row has no stored
    probabilities: it contributes nothing (and checked mode reports it)."""
    wl, H, W, y = _case(400, 128, 3000, seed=5)
    m = (np.arange(400) % 4 != 0)
    mask = torch.as_tensor(m.astype(np.uint8)).cuda()
    cache = sao.logprob_cache(400, 3000)
    logp, lse = _fwd(H, W, y, cache, row_mask=mask)
    G = np.random.default_rng(9).normal(size=400).astype(np.float32)
    G_masked = np.where(m, G, 0).astype(np.float32)
    dH, dW = _bwd(H, W, y, lse, torch.as_tensor(G_masked).cuda(), cache)
    torch.cuda.synchronize()
    want_lp, want_lse = O.token_logprobs(H.cpu(), W.cpu(), wl.y)
    got = logp.cpu().numpy()
    assert np.all(got[~m] == 0) and np.abs(got[m] - want_lp[m]).max() <= LOGP_TOL
    want_dH, want_dW = O.token_logprobs_bwd(H.cpu(), W.cpu(), wl.y, want_lse, G_masked)
    assert rel_l2(dH.float().cpu().numpy(), want_dH) <= GRAD_TOL
    assert rel_l2(dW.cpu().numpy(), want_dW) <= GRAD_TOL
    # unchecked: rows the forward skipped drop out of the gradient
    dH2, dW2 = _bwd(H, W, y, lse, torch.as_tensor(G).cuda(), cache)
    torch.cuda.synchronize()
    assert rel_l2(dW2.cpu().numpy(), want_dW) <= GRAD_TOL
    assert not dH2.float().cpu().numpy()[~m].any()
    sao.sao_set_checked(True)
    try:
        with pytest.raises(sao.SaoError) as e:
            _bwd(H, W, y, lse, torch.as_tensor(G).cuda(), cache)
        assert e.value.status == 6
    finally:
        sao.sao_set_checked(False)


def test_cached_forward_with_every_row_skipped():
    """A row mask of zeros leaves no forward row: log-probs are 0, and a
    backward with a zero gradient writes zeros to dH and dW, or leaves an
    accumulated dW as it was."""
    wl, H, W, y = _case(300, 64, 1000, seed=23)
    mask = torch.zeros(300, dtype=torch.uint8, device="cuda")
    cache = sao.logprob_cache(300, 1000)
    logp, lse = _fwd(H, W, y, cache, row_mask=mask)
    G = torch.zeros(300, device="cuda")
    dH, dW = _bwd(H, W, y, lse, G, cache)
    prev = torch.randn(1000, 64, device="cuda")
    dH2, dW2 = _bwd(H, W, y, lse, G, cache, accumulate=prev)
    torch.cuda.synchronize()
    assert not logp.cpu().numpy().any() and not lse.cpu().numpy().any()
    assert not dH.float().cpu().numpy().any() and not dW.cpu().numpy().any()
    assert not dH2.float().cpu().numpy().any()
    assert torch.equal(dW2, prev)


def test_cached_backward_chunked_and_accumulate():
    """A small dZ budget forces several vocabulary chunks (the last one ragged,
    not a multiple of 8 columns); accumulate_dW adds to dW."""
    wl, H, W, y = _case(700, 128, 3003, seed=19)
    cache = sao.logprob_cache(700, 3003)
    logp, lse = _fwd(H, W, y, cache)
    G = np.random.default_rng(3).normal(size=700).astype(np.float32)
    prev = torch.randn(3003, 128, device="cuda")
    sao.sao_set_dz_budget_bytes(700 * 512 * 2)       # one row block, Vc = 512: 6 vocabulary chunks
    try:
        dH, dW = _bwd(H, W, y, lse, torch.as_tensor(G).cuda(), cache, accumulate=prev)
        torch.cuda.synchronize()
    finally:
        sao.sao_set_dz_budget_bytes(DEFAULT_DZ_BUDGET)
    _, want_lse = O.token_logprobs(H.cpu(), W.cpu(), wl.y)
    want_dH, want_dW = O.token_logprobs_bwd(H.cpu(), W.cpu(), wl.y, want_lse, G)
    assert rel_l2(dH.float().cpu().numpy(), want_dH) <= GRAD_TOL
    assert rel_l2(dW.cpu().numpy() - prev.cpu().numpy(), want_dW) <= GRAD_TOL


def test_cached_moe_bench_configuration_sampled_rows():
    """The moe step as bench.py runs it (row_mask = loss_mask, gradient on
    action rows): logp, lse and dH on sampled rows, dW on sampled vocabulary
    rows, against the oracle's own forward on those rows."""
    wl = S.make_workload("moe", device="cuda")
    N, h, V = wl.N, wl.h, wl.V
    y = torch.as_tensor(wl.y).cuda()
    mask = torch.as_tensor(wl.loss_mask).cuda()
    cache = sao.logprob_cache(N, V)
    logp, lse = _fwd(wl.H, wl.W, y, cache, row_mask=mask)
    rng = np.random.default_rng(14)
    act = np.flatnonzero(wl.loss_mask)
    rows = np.sort(rng.choice(act, size=32, replace=False))
    G = np.zeros(N, np.float32)
    G[rows] = rng.normal(size=len(rows)).astype(np.float32)
    dH, dW = _bwd(wl.H, wl.W, y, lse, torch.as_tensor(G).cuda(), cache)
    torch.cuda.synchronize()
    H_cpu, W_cpu = wl.H[torch.as_tensor(rows).cuda()].cpu(), wl.W.cpu()
    want_lp, want_lse = O.token_logprobs(H_cpu, W_cpu, wl.y[rows])
    assert np.abs(logp.cpu().numpy()[rows] - want_lp).max() <= LOGP_TOL
    want_dH, _ = O.token_logprobs_bwd(H_cpu, W_cpu, wl.y[rows], want_lse, G[rows])
    got_dH = dH.float().cpu().numpy()
    assert rel_l2(got_dH[rows], want_dH) <= GRAD_TOL
    others = np.ones(N, bool)
    others[rows] = False
    assert not np.any(got_dH[others])
    vrows = np.unique(np.concatenate([rng.choice(V, size=512, replace=False), wl.y[rows], [V - 1]]))
    Wsub = W_cpu[torch.as_tensor(vrows)]
    pos = {int(v): i for i, v in enumerate(vrows)}
    Hd = O._f64(H_cpu)
    dZ = -G[rows].astype(np.float64)[:, None] * np.exp(Hd @ O._f64(Wsub).T - want_lse[:, None])
    for i, t in enumerate(wl.y[rows]):
        j = pos.get(int(t), -1)
        if j >= 0:
            dZ[i, j] += G[rows][i]
    want_dW = dZ.T @ Hd
    got_dW = dW[torch.as_tensor(vrows).cuda()].cpu().numpy()
    assert rel_l2(got_dW, want_dW) <= GRAD_TOL


@pytest.mark.parametrize("cached,chunked", [(True, False), (False, False), (True, True)])
def test_two_m_tile_gemms_with_ragged_tiles(cached, chunked):
    """A shape at which both backward GEMMs take two 128-row M tiles per CTA
    tile (at least four waves of paired tiles on the GPU): 20,100 rows and
    20,168 vocabulary rows, so the last paired tile of dW has a full first and
    a 72-row second tile, and dH's last pair a partial first tile only. With
    `chunked` a small dZ budget splits the vocabulary into chunks, so dH
    accumulates in fp32 (the other store epilogue) and is scattered at the end.
    logp, dH on sampled rows and dW on sampled vocabulary rows (the last 72
    included) against the oracle."""
    N, h, V = 20100, 2048, 20168
    wl = S.make_custom([N], h, V, "bf16", seed=77, device="cuda")
    H, W, y = wl.H, wl.W, torch.as_tensor(wl.y).cuda()
    ws = sao.workspace(N, h, V, H.dtype)
    logp = torch.empty(N, device="cuda")
    lse = torch.empty(N, device="cuda")
    rng = np.random.default_rng(78)
    G = rng.normal(size=N).astype(np.float32)
    G[rng.random(N) < 0.01] = 0.0
    Gd = torch.as_tensor(G).cuda()
    dH = torch.full_like(H, float("nan"))
    dW = torch.full((V, h), float("nan"), device="cuda")
    if chunked:
        sao.sao_set_dz_budget_bytes(N * 5120 * 2)       # several vocabulary chunks, the last one ragged
    try:
        if cached:
            cache = sao.logprob_cache(N, V)
            sao.sao_token_logprobs_fwd_cached(H, W, y, logp, lse, cache, ws)
            sao.sao_token_logprobs_bwd_cached(H, W, y, lse, Gd, dH, dW, cache, ws)
        else:
            sao.sao_token_logprobs_fwd(H, W, y, logp, lse, ws)
            sao.sao_token_logprobs_bwd(H, W, y, lse, Gd, dH, dW, ws)
        torch.cuda.synchronize()
    finally:
        if chunked:
            sao.sao_set_dz_budget_bytes(DEFAULT_DZ_BUDGET)
    rows = np.sort(np.concatenate([rng.choice(N, size=24, replace=False), [N - 1]]))
    H_cpu, W_cpu = H[torch.as_tensor(rows).cuda()].cpu(), W.cpu()
    want_lp, want_lse = O.token_logprobs(H_cpu, W_cpu, wl.y[rows])
    assert np.abs(logp.cpu().numpy()[rows] - want_lp).max() <= LOGP_TOL
    want_dH, _ = O.token_logprobs_bwd(H_cpu, W_cpu, wl.y[rows], want_lse, G[rows])
    assert rel_l2(dH.float().cpu().numpy()[rows], want_dH) <= GRAD_TOL
    # dW rows: every token contributes; the GPU lse (checked on the sampled rows) stands in for the
    # full-vocabulary lse of all 20,100 rows
    vrows = np.unique(np.concatenate([rng.choice(V, size=48, replace=False), np.arange(V - 72, V)]))
    Hd = O._f64(H.cpu())
    Z = Hd @ O._f64(W_cpu[torch.as_tensor(vrows)]).T                       # [N, |vrows|]
    lse_gpu = lse.cpu().numpy().astype(np.float64)                           # the forward's lse (checked above)
    dZ = -G.astype(np.float64)[:, None] * np.exp(Z - lse_gpu[:, None])
    pos = {int(v): i for i, v in enumerate(vrows)}
    for t in range(N):
        j = pos.get(int(wl.y[t]), -1)
        if j >= 0:
            dZ[t, j] += G[t]
    want_dW = dZ.T @ Hd
    got_dW = dW[torch.as_tensor(vrows).cuda()].cpu().numpy()
    assert rel_l2(got_dW, want_dW) <= GRAD_TOL


def test_cached_argument_errors():
    wl, H, W, y = _case(64, 64, 300, seed=3)
    logp = torch.empty(64, device="cuda")
    lse = torch.empty(64, device="cuda")
    ws = sao.workspace(64, 64, 300, H.dtype)
    small = torch.empty(sao.sao_logprob_cache_bytes(64, 300) - 256, dtype=torch.uint8, device="cuda")
    with pytest.raises(sao.SaoError) as e:
        sao.sao_token_logprobs_fwd_cached(H, W, y, logp, lse, small, ws)
    assert e.value.status == 3
    big = torch.empty(sao.sao_logprob_cache_bytes(64, 300) + 512, dtype=torch.uint8, device="cuda")
    with pytest.raises(sao.SaoError) as e:
        sao.sao_token_logprobs_fwd_cached(H, W, y, logp, lse, big[16:], ws)
    assert e.value.status == 1
    Hf, Wf = H.float(), W.float()
    with pytest.raises(sao.SaoError) as e:
        sao.sao_token_logprobs_fwd_cached(Hf, Wf, y, logp, lse, big, sao.workspace(64, 64, 300, torch.float32))
    assert e.value.status == 4


@pytest.mark.parametrize("chunked,masked", [(False, False), (True, True), (False, True)])
def test_cached_rows_far_below_their_maximum_are_recomputed(chunked, masked):
    """Rows whose sampled token's logit lies 64 nats below another logit of the
    row exceed the stored range (e relative to the sampled token's logit):
    the forward flags them and still returns their exact lse and log-prob,
    and the backward recomputes their logits. One flagged row has a zero
    gradient (nothing to recompute), one unflagged row shares its token.
    chunked: a small dZ budget makes the recompute run in vocabulary chunks
    (fp32 dH accumulator, then a scatter of the flagged rows only) and dW
    accumulates onto given contents; masked: a row mask skips some rows, so
    forward rows and tokens are numbered differently."""
    N, h, V = 300, 64, 1000
    wl, H, W, y = _case(N, h, V, seed=41)
    H, W = H.clone(), W.clone()
    yv = wl.y.copy()
    jstar = 7
    far = [5, 130, 299, 200]
    for r in far:
        yv[r] = 11 + r
        H[r].zero_()
        H[r, 0] = 8.0
        W[11 + r].zero_()
        W[11 + r, 0] = -4.0   # z[r, y] = -32
    W[jstar].zero_()
    W[jstar, 0] = 4.0         # z[r, jstar] = +32: 64 nats above the sampled token
    yv[17] = 11 + 5           # an ordinary row sampling the same token
    y = torch.as_tensor(yv).cuda()
    rng = np.random.default_rng(43)
    G = rng.normal(size=N).astype(np.float32)
    G[200] = 0.0
    mask = None
    if masked:
        m = (rng.random(N) < 0.7).astype(np.uint8)
        m[far] = 1
        m[17] = 1
        G[m == 0] = 0.0
        mask = torch.as_tensor(m).cuda()
    cache = sao.logprob_cache(N, V)
    logp, lse = _fwd(H, W, y, cache, row_mask=mask)
    prev = torch.randn(V, h, device="cuda") if chunked else None
    if chunked:
        sao.sao_set_dz_budget_bytes(N * 256 * 2)     # several vocabulary chunks, the last ragged
    try:
        dH, dW = _bwd(H, W, y, lse, torch.as_tensor(G).cuda(), cache, accumulate=prev)
        torch.cuda.synchronize()
    finally:
        sao.sao_set_dz_budget_bytes(DEFAULT_DZ_BUDGET)
    want_lp, want_lse = O.token_logprobs(H.cpu(), W.cpu(), yv)
    assert want_lp[far].max() < -60.0
    got_lp, got_lse = logp.cpu().numpy(), lse.cpu().numpy()
    keep = np.ones(N, bool) if mask is None else mask.cpu().numpy() != 0
    assert np.abs(got_lp[keep] - want_lp[keep]).max() <= LOGP_TOL
    assert np.abs(got_lse[keep] - want_lse[keep]).max() <= LOGP_TOL
    want_dH, want_dW = O.token_logprobs_bwd(H.cpu(), W.cpu(), yv, want_lse, G)
    got_dH = dH.float().cpu().numpy()
    got_dW = dW.cpu().numpy() - (prev.cpu().numpy() if chunked else 0.0)
    assert rel_l2(got_dH, want_dH) <= GRAD_TOL
    for r in far:
        if G[r] == 0:
            assert np.all(got_dH[r] == 0)
        else:
            assert rel_l2(got_dH[r], want_dH[r]) <= GRAD_TOL
    assert np.all(got_dH[G == 0] == 0)
    assert rel_l2(got_dW, want_dW) <= GRAD_TOL
    assert np.all(np.isfinite(got_dW))
