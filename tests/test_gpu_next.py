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


def test_step_advantages_no_action_tokens():
    wl = S.make_custom([10, 300], 8, 16, "f32", seed=4, dense=False)
    wl.loss_mask[:] = 0
    adv, ret, vm = _step_gpu(wl, 1.0, 1.0, 1.0, 0.0, sao.SAO_STEP_AVERAGE)
    assert not adv.any() and not ret.any() and not vm.any()
