"""sao_advantages_noalloc: the advantage scan for callers that cannot allocate
device memory (it uses the library's fixed device scratch instead of a
workspace). Called through the C ABI, twice in a row on different batches,
and compared with sao_advantages given a workspace. Collected last so that a
run stopping at its first failure has already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2607_07508_gb300 import sao, synthetic as S
from tests._util import rel_err_floor

pytestmark = pytest.mark.gpu

ADV_TOL = 1e-5  # relative to max(|A|, 1e-3), as for sao_advantages


def _with_workspace(wl, args):
    adv = torch.empty(wl.N, device="cuda")
    ret = torch.empty(wl.N, device="cuda")
    sao.sao_advantages(*args, adv, ret, sao.workspace(wl.N))
    return adv, ret


def _no_alloc(wl, args):
    adv = torch.full((wl.N,), float("nan"), device="cuda")
    ret = torch.full((wl.N,), float("nan"), device="cuda")
    sao.sao_advantages_noalloc(*args, adv, ret)
    return adv, ret


@pytest.mark.parametrize("order", [("moe", "long"), ("long", "moe")])
def test_no_alloc_matches_workspace_entry_point(order):
    for name in order:            # two calls in a row share the static scratch
        wl = S.make_workload(name, dense=False)
        args = [torch.as_tensor(a).cuda() for a in (wl.values, wl.rewards, wl.loss_mask, wl.cu_seqlens)]
        args += [wl.gamma, wl.lam, wl.lam_critic, wl.alpha]
        a0, r0 = _with_workspace(wl, args)
        a1, r1 = _no_alloc(wl, args)
        torch.cuda.synchronize()
        a0, r0, a1, r1 = (t.cpu().numpy() for t in (a0, r0, a1, r1))
        assert rel_err_floor(a1, a0, 1e-3).max() <= ADV_TOL
        assert rel_err_floor(r1, r0, 1e-3).max() <= ADV_TOL


def test_no_alloc_rejects_sizes_beyond_its_scratch():
    lib = sao.load()
    P = ctypes.c_void_p(16)
    st = lib.sao_advantages_noalloc(P, P, P, P, 1 << 22, (1 << 31) - 1, 1.0, 1.0, 1.0, 0.0, P, P, None)
    assert st == 2
    assert "scratch" in lib.sao_last_error_string().decode()


def test_no_alloc_documented_example_fits():
    """The size the header quotes (2^25 tokens in 65,536 trajectories) fits
    the fixed scratch and matches the workspace entry point."""
    N, B = 1 << 25, 1 << 16
    rng = np.random.default_rng(21)
    cu = np.arange(0, N + 1, N // B, dtype=np.int32)
    values = rng.standard_normal(N, dtype=np.float32)
    mask = (rng.random(N) < 0.75).astype(np.uint8)
    rewards = (rng.random(B) < 0.4).astype(np.float32)
    args = [torch.as_tensor(a).cuda() for a in (values, rewards, mask, cu)] + [1.0, 0.95, 1.0, 0.0]

    class _Shape:
        pass
    wl = _Shape()
    wl.N = N
    a0, r0 = _with_workspace(wl, args)
    a1, r1 = _no_alloc(wl, args)
    torch.cuda.synchronize()
    assert torch.equal(a0, a1) and torch.equal(r0, r1)
