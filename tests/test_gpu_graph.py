"""The loss-head step captured into a CUDA graph. Every entry point is
asynchronous on its stream and never synchronises the host (checked mode off),
workspaces are zeroed by the calls themselves, and every reduction and scan
gives the same bits whatever the timing, so a captured step replays to exactly
the eager results. The first eager call sets up the library's per-process
state (function attributes, device properties) before the capture."""
import numpy as np
import pytest
import torch

from paper_2607_07508_gb300 import sao, synthetic as S
from tests._util import cuda

pytestmark = pytest.mark.gpu


def _buffers(wl):
    N, h, V = wl.N, wl.h, wl.V
    f = lambda: torch.empty(N, device="cuda")
    b = {"y": cuda(wl.y), "m": cuda(wl.loss_mask), "v": cuda(wl.values), "R": cuda(wl.rewards),
         "cu": cuda(wl.cu_seqlens), "adv": f(), "ret": f(), "dV": f(), "logp": f(), "lse": f(), "coef": f(),
         "G": f(), "vloss": torch.empty(1, device="cuda"), "loss": torch.empty(1, device="cuda"),
         "counts": torch.empty(4, dtype=torch.int64, device="cuda"),
         "flags": torch.empty(N, dtype=torch.uint8, device="cuda"), "one": torch.ones(1, device="cuda"),
         "dH": torch.empty_like(wl.H), "dW": torch.empty(V, h, device="cuda"),
         "ws": sao.workspace(N, h, V, wl.H.dtype), "cache": sao.logprob_cache(N, V)}
    lp = torch.empty(N, device="cuda")
    lse = torch.empty(N, device="cuda")
    sao.sao_token_logprobs_fwd(wl.H, wl.W, b["y"], lp, lse, b["ws"])
    b["old"] = (lp + cuda(wl.xi)).contiguous()
    return b


def _step(wl, b):
    sao.sao_advantages(b["v"], b["R"], b["m"], b["cu"], wl.gamma, wl.lam, wl.lam_critic, wl.alpha, b["adv"],
                       b["ret"], b["ws"])
    sao.sao_value_loss(b["v"], b["ret"], b["m"], b["vloss"], b["dV"], b["ws"])
    sao.sao_token_logprobs_fwd_cached(wl.H, wl.W, b["y"], b["logp"], b["lse"], b["cache"], b["ws"], row_mask=b["m"])
    sao.sao_policy_loss_fwd(b["logp"], b["old"], b["adv"], b["m"], wl.eps_low, wl.eps_high, b["loss"], b["counts"],
                            b["ws"], coef=b["coef"], flags=b["flags"])
    sao.sao_policy_loss_bwd(b["logp"], b["old"], b["adv"], b["m"], wl.eps_low, wl.eps_high, b["one"], b["G"],
                            b["ws"])
    sao.sao_token_logprobs_bwd_cached(wl.H, wl.W, b["y"], b["lse"], b["G"], b["dH"], b["dW"], b["cache"], b["ws"])


OUTPUTS = ("adv", "ret", "dV", "vloss", "logp", "lse", "loss", "counts", "coef", "flags", "G", "dH", "dW")


def test_captured_step_replays_bit_identically():
    wl = S.make_workload("small", device="cuda")
    b = _buffers(wl)
    _step(wl, b)
    torch.cuda.synchronize()
    eager = {k: b[k].clone() for k in OUTPUTS}
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        _step(wl, b)
    for _ in range(2):
        for k in OUTPUTS:                      # poison the outputs: the replay must rewrite them
            if b[k].dtype.is_floating_point:
                b[k].fill_(float("nan"))
            else:
                b[k].fill_(-1 if b[k].dtype == torch.int64 else 9)
        graph.replay()
        torch.cuda.synchronize()
        for k in OUTPUTS:
            assert torch.equal(b[k], eager[k]), k


def test_advantage_scan_is_bit_identical_at_scale():
    """2^24 tokens in ~2,500 trajectories: thousands of chunks whose look-backs
    race each other; three runs give the same bits."""
    wl = S.bandwidth_workload(N=1 << 24, B=1 << 11)
    v, m, cu, R = (cuda(x) for x in (wl.values, wl.loss_mask, wl.cu_seqlens, wl.rewards))
    ws = sao.workspace(wl.N)
    outs = []
    for gamma, lam, lam_c, alpha in ((1.0, 0.95, 1.0, 0.0), (0.99, 0.9, 0.97, 1.5)):
        for _ in range(3):
            adv = torch.empty(wl.N, device="cuda")
            ret = torch.empty(wl.N, device="cuda")
            sao.sao_advantages(v, R, m, cu, gamma, lam, lam_c, alpha, adv, ret, ws)
            outs.append((adv, ret))
        torch.cuda.synchronize()
        a0, r0 = outs[-3]
        for a, r in outs[-2:]:
            assert torch.equal(a, a0) and torch.equal(r, r0)
        assert np.isfinite(a0.cpu().numpy()).all()
