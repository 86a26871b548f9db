"""GPU parity of the LM-head log-probs (Eq. 1-2) and their gradient with the
fp64 oracle through the C ABI: bf16 tensor-core path (tcgen05) and fp32 path,
on shapes that span several 128x256 tiles with ragged tails in every
dimension, plus edge cases (V = 1, N = 1, masked rows, zero gradients,
vocabulary chunking, accumulation into dW)."""
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


def _fwd(H, W, y, row_mask=None):
    N, h = H.shape
    V = W.shape[0]
    logp = torch.empty(N, device="cuda")
    lse = torch.empty(N, device="cuda")
    ws = sao.workspace(N, h, V, H.dtype)
    sao.sao_token_logprobs_fwd(H, W, y, logp, lse, ws, row_mask=row_mask)
    return logp, lse


def _bwd(H, W, y, lse, G, accumulate=None):
    N, h = H.shape
    V = W.shape[0]
    dH = torch.empty_like(H)
    dW = accumulate.clone() if accumulate is not None else torch.empty(V, h, device="cuda")
    ws = sao.workspace(N, h, V, H.dtype)
    sao.sao_token_logprobs_bwd(H, W, y, lse, G, dH, dW, ws, accumulate_dW=accumulate is not None)
    return dH, dW


def _case(N, h, V, dtype, seed):
    wl = S.make_custom([N], h, V, dtype, seed=seed, device="cuda")
    y = torch.as_tensor(wl.y).cuda()
    return wl, wl.H, wl.W, y


CASES = [(300, 192, 1000, "bf16"), (1000, 256, 4113, "bf16"), (129, 64, 257, "bf16"), (1, 8, 1, "bf16"),
         (513, 520, 2000, "bf16"), (77, 40, 300, "f32"), (1169, 256, 4096, "f32"), (2, 16, 1, "f32")]


@pytest.mark.parametrize("N,h,V,dt", CASES)
def test_logprobs_forward(N, h, V, dt):
    wl, H, W, y = _case(N, h, V, dt, seed=N + h + V)
    logp, lse = _fwd(H, W, y)
    torch.cuda.synchronize()
    want_lp, want_lse = O.token_logprobs(H.cpu(), W.cpu(), wl.y)
    assert np.abs(logp.cpu().numpy() - want_lp).max() <= LOGP_TOL
    assert np.abs(lse.cpu().numpy() - want_lse).max() <= LOGP_TOL


@pytest.mark.parametrize("N,h,V,dt", CASES)
def test_logprobs_backward(N, h, V, dt):
    wl, H, W, y = _case(N, h, V, dt, seed=N + h + V)
    logp, lse = _fwd(H, W, y)
    rng = np.random.default_rng(N)
    G = rng.normal(size=N).astype(np.float32)
    G[rng.random(N) < 0.3] = 0.0
    Gt = torch.as_tensor(G).cuda()
    dH, dW = _bwd(H, W, y, lse, Gt)
    torch.cuda.synchronize()
    _, want_lse = O.token_logprobs(H.cpu(), W.cpu(), wl.y)
    want_dH, want_dW = O.token_logprobs_bwd(H.cpu(), W.cpu(), wl.y, want_lse, G)
    assert rel_l2(dH.float().cpu().numpy(), want_dH) <= GRAD_TOL
    assert rel_l2(dW.cpu().numpy(), want_dW) <= GRAD_TOL
    zero_rows = G == 0
    assert np.all(dH.float().cpu().numpy()[zero_rows] == 0)


def test_logprobs_row_mask_and_bad_token():
    wl, H, W, y = _case(300, 64, 700, "bf16", seed=1)
    mask = torch.as_tensor((np.arange(300) % 3 != 0).astype(np.uint8)).cuda()
    logp, lse = _fwd(H, W, y, row_mask=mask)
    torch.cuda.synchronize()
    want_lp, _ = O.token_logprobs(H.cpu(), W.cpu(), wl.y)
    got = logp.cpu().numpy()
    m = mask.cpu().numpy().astype(bool)
    assert np.all(got[~m] == 0) and np.abs(got[m] - want_lp[m]).max() <= LOGP_TOL
    y2 = y.clone()
    y2[5] = 700
    sao.sao_set_checked(True)
    try:
        with pytest.raises(sao.SaoError) as e:
            _fwd(H, W, y2)
        assert e.value.status == 6
    finally:
        sao.sao_set_checked(False)
    logp, _ = _fwd(H, W, y2)
    assert np.isnan(logp[5].item())


def test_logprobs_backward_chunked_and_accumulate():
    """A small dZ budget forces several vocabulary chunks and the fp32 dH
    accumulator; accumulate_dW adds to the previous contents of dW."""
    wl, H, W, y = _case(700, 128, 3000, "bf16", seed=9)
    logp, lse = _fwd(H, W, y)
    G = np.random.default_rng(3).normal(size=700).astype(np.float32)
    prev = torch.randn(3000, 128, device="cuda")
    sao.sao_set_dz_budget_bytes(700 * 512 * 2)       # one row block, Vc = 512: 6 vocabulary chunks
    try:
        dH, dW = _bwd(H, W, y, lse, torch.as_tensor(G).cuda(), accumulate=prev)
        torch.cuda.synchronize()
    finally:
        sao.sao_set_dz_budget_bytes(DEFAULT_DZ_BUDGET)
    _, want_lse = O.token_logprobs(H.cpu(), W.cpu(), wl.y)
    want_dH, want_dW = O.token_logprobs_bwd(H.cpu(), W.cpu(), wl.y, want_lse, G)
    assert rel_l2(dH.float().cpu().numpy(), want_dH) <= GRAD_TOL
    assert rel_l2(dW.cpu().numpy() - prev.cpu().numpy(), want_dW) <= GRAD_TOL


def test_tiny_config_full_oracle():
    wl = S.make_workload("tiny", device="cuda")
    y = torch.as_tensor(wl.y).cuda()
    logp, lse = _fwd(wl.H, wl.W, y)
    G = np.random.default_rng(4).normal(size=wl.N).astype(np.float32) * 1e-3
    dH, dW = _bwd(wl.H, wl.W, y, lse, torch.as_tensor(G).cuda())
    torch.cuda.synchronize()
    want_lp, want_lse = O.token_logprobs(wl.H.cpu(), wl.W.cpu(), wl.y)
    assert np.abs(logp.cpu().numpy() - want_lp).max() <= LOGP_TOL
    want_dH, want_dW = O.token_logprobs_bwd(wl.H.cpu(), wl.W.cpu(), wl.y, want_lse, G)
    assert rel_l2(dH.cpu().numpy(), want_dH) <= GRAD_TOL
    assert rel_l2(dW.cpu().numpy(), want_dW) <= GRAD_TOL


@pytest.mark.parametrize("dt", ["bf16", "f32"])
def test_logprobs_backward_all_zero_gradient(dt):
    """No active row: dH = 0, dW = 0 (or unchanged when accumulating)."""
    wl, H, W, y = _case(300, 64, 700, dt, seed=2)
    logp, lse = _fwd(H, W, y)
    G = torch.zeros(300, device="cuda")
    dH, dW = _bwd(H, W, y, lse, G)
    prev = torch.randn(700, 64, device="cuda")
    _, dW2 = _bwd(H, W, y, lse, G, accumulate=prev)
    torch.cuda.synchronize()
    assert not dH.float().abs().max().item() and not dW.abs().max().item()
    assert torch.equal(dW2, prev)


def test_logprobs_backward_all_zero_gradient_paired_tiles():
    """The same with h = 2048 and V = 20,000, where the dW GEMM takes two M
    tiles per CTA tile: the empty contraction writes zeros to both tiles, or
    leaves dW unchanged when accumulating; on both log-prob paths."""
    wl, H, W, y = _case(300, 2048, 20000, "bf16", seed=4)
    logp, lse = _fwd(H, W, y)
    G = torch.zeros(300, device="cuda")
    dH, dW = _bwd(H, W, y, lse, G)
    prev = torch.randn(20000, 2048, device="cuda")
    _, dW2 = _bwd(H, W, y, lse, G, accumulate=prev)
    cache = sao.logprob_cache(300, 20000)
    ws = sao.workspace(300, 2048, 20000, H.dtype)
    sao.sao_token_logprobs_fwd_cached(H, W, y, logp, lse, cache, ws)
    dH3 = torch.full_like(H, float("nan"))
    dW3 = torch.full((20000, 2048), float("nan"), device="cuda")
    sao.sao_token_logprobs_bwd_cached(H, W, y, lse, G, dH3, dW3, cache, ws)
    torch.cuda.synchronize()
    assert not dH.float().abs().max().item() and not dW.abs().max().item()
    assert torch.equal(dW2, prev)
    assert not dH3.float().abs().max().item() and not dW3.abs().max().item()
