"""ABI contract on the GPU: determinism, stream semantics, error paths."""
import numpy as np
import pytest
import torch

from paper_2607_07508_gb300 import sao, synthetic as S
from tests._util import cuda

pytestmark = pytest.mark.gpu


def _step(wl, stream=None):
    """All six calls on one stream; returns every output."""
    N, h, V = wl.N, wl.h, wl.V
    dev = "cuda"
    out = {}
    with torch.cuda.stream(stream) if stream is not None else torch.cuda.stream(torch.cuda.current_stream()):
        y, m = cuda(wl.y), cuda(wl.loss_mask)
        vals, R, cu = cuda(wl.values), cuda(wl.rewards), cuda(wl.cu_seqlens)
        ws = sao.workspace(N, h, V, wl.H.dtype)
        f = lambda: torch.empty(N, device=dev)
        out["adv"], out["ret"] = f(), f()
        sao.sao_advantages(vals, R, m, cu, wl.gamma, wl.lam, wl.lam_critic, wl.alpha, out["adv"], out["ret"], ws)
        out["vloss"] = torch.empty(1, device=dev)
        out["dV"] = f()
        sao.sao_value_loss(vals, out["ret"], m, out["vloss"], out["dV"], ws)
        out["logp"], out["lse"] = f(), f()
        sao.sao_token_logprobs_fwd(wl.H, wl.W, y, out["logp"], out["lse"], ws, row_mask=m)
        old = (out["logp"] + cuda(wl.xi)).contiguous()
        out["loss"] = torch.empty(1, device=dev)
        out["counts"] = torch.empty(4, dtype=torch.int64, device=dev)
        sao.sao_policy_loss_fwd(out["logp"], old, out["adv"], m, wl.eps_low, wl.eps_high, out["loss"],
                                out["counts"], ws)
        out["G"] = f()
        sao.sao_policy_loss_bwd(out["logp"], old, out["adv"], m, wl.eps_low, wl.eps_high,
                                torch.ones(1, device=dev), out["G"], ws)
        out["dH"] = torch.empty_like(wl.H)
        out["dW"] = torch.empty(V, h, device=dev)
        sao.sao_token_logprobs_bwd(wl.H, wl.W, y, out["lse"], out["G"], out["dH"], out["dW"], ws)
    torch.cuda.synchronize()
    return {k: v.cpu() for k, v in out.items()}


def test_step_is_deterministic_and_stream_independent():
    """Two runs on the default stream and one on a side stream give bit-identical
    outputs (fixed-order reductions, no atomics on the data path)."""
    wl = S.make_custom([700, 0, 1500, 333], 256, 5000, "bf16", seed=31, device="cuda", obs_frac=0.25)
    a = _step(wl)
    b = _step(wl)
    c = _step(wl, torch.cuda.Stream())
    for k in a:
        assert torch.equal(a[k], b[k]), k
        assert torch.equal(a[k], c[k]), k


def test_misaligned_bf16_operand_is_rejected():
    """TMA needs 16-byte aligned operands: an offset H view is refused with an
    argument error, not launched."""
    wl = S.make_custom([64], 64, 300, "bf16", seed=1, device="cuda")
    H = torch.empty(65 * 64, dtype=torch.bfloat16, device="cuda")[1:1 + 64 * 64].view(64, 64)
    H.copy_(wl.H)
    logp = torch.empty(64, device="cuda")
    lse = torch.empty(64, device="cuda")
    with pytest.raises(sao.SaoError) as e:
        sao.sao_token_logprobs_fwd(H, wl.W, cuda(wl.y), logp, lse, sao.workspace(64, 64, 300))
    assert e.value.status == 1


def test_small_workspace_is_rejected():
    wl = S.make_custom([64], 64, 300, "bf16", seed=1, device="cuda")
    ws = torch.empty(1024, dtype=torch.uint8, device="cuda")
    with pytest.raises(sao.SaoError) as e:
        sao.sao_token_logprobs_fwd(wl.H, wl.W, cuda(wl.y), torch.empty(64, device="cuda"),
                                   torch.empty(64, device="cuda"), ws)
    assert e.value.status == 3
