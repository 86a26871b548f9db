"""Failure detection on the GPU without a fault. The advantage scan's bounded
look-back wait is made to run out through its test hooks (a short wait limit
and top chunks that are never processed: a carry that nothing publishes). The
call still completes, checked mode reports the time-out through the device
error word, and the context stays usable: the next call is correct."""
import time

import numpy as np
import pytest
import torch

from oracle import sao_oracle as O
from paper_2607_07508_gb300 import sao, synthetic as S
from tests._util import cuda, rel_err_floor

pytestmark = pytest.mark.gpu


def test_scan_wait_runs_out_and_is_reported():
    wl = S.make_custom([8192] * 8, 8, 16, "f32", seed=5, dense=False, obs_frac=0.3)
    N = wl.N
    args = [cuda(x) for x in (wl.values, wl.rewards, wl.loss_mask, wl.cu_seqlens)] + [1.0, 0.95, 1.0, 0.0]
    adv = torch.empty(N, device="cuda")
    ret = torch.empty(N, device="cuda")
    ws = sao.workspace(N)
    sao.sao_debug_set_scan_hooks(20_000_000, 3)   # 20 ms waits; the top 3 chunks never run
    sao.sao_set_checked(True)
    try:
        t0 = time.time()
        with pytest.raises(sao.SaoError) as e:
            sao.sao_advantages(*args, adv, ret, ws)
        assert e.value.status == 6
        assert "scan-carry-timeout" in str(e.value)
        assert time.time() - t0 < 30
    finally:
        sao.sao_debug_set_scan_hooks(0, 0)
        sao.sao_set_checked(False)
    # the context is intact: the same call succeeds in checked mode and is right
    sao.sao_set_checked(True)
    try:
        sao.sao_advantages(*args, adv, ret, ws)
    finally:
        sao.sao_set_checked(False)
    torch.cuda.synchronize()
    want_a, want_r = O.advantages(wl.values, wl.rewards, wl.loss_mask, wl.cu_seqlens, 1.0, float(np.float32(0.95)),
                                  1.0, 0.0)
    assert rel_err_floor(adv.cpu().numpy(), want_a, 1e-3).max() <= 1e-5
    assert rel_err_floor(ret.cpu().numpy(), want_r, 1e-3).max() <= 1e-5
