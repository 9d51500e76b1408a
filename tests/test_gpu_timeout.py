"""The bounded device wait and its status bit, without a fault.

The separate hidden ranking stages the query row H_{t-1} in shared memory with a
bulk copy and waits for it with a bounded mbarrier wait; when the wait runs out
the sequence gets PLDP_ST_TIMEOUT and no choice, and the call returns.  To make
the wait run out without breaking anything, a test build of the ranking
(PLDP_TEST_STUCK_QUERY_WAIT) has its scoring warps wait on a barrier that nothing
arrives on, with a short bound; the copy itself still lands, and each CTA waits
for it before it exits.  The test then checks the status, the outputs and that
the CUDA context is still usable."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2412_01447_gb300 import _build

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _stuck_lib():
    path = _build.build_variant("stuck_query_wait", ["rank.cu", "abi.cu"],
                                extra_flags=["-DPLDP_TEST_STUCK_QUERY_WAIT"])
    lib = ctypes.CDLL(path)
    P, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
    lib.pldp_rank_hidden.argtypes = [P, i32, i64, i64, P, i32, i64, P, P, i32, ctypes.c_float, P, P, P, P, P]
    lib.pldp_rank_hidden.restype = i32
    return lib


@pytest.mark.parametrize("B,C_cap", [(4, 4), (6, 80)])      # one CTA per candidate; warps on their own
def test_query_wait_runs_out(lib, B, C_cap):
    stuck = _stuck_lib()
    T, d = 96, 512
    H = torch.randn((B, T, d), device=DEV).to(torch.bfloat16)
    rng = np.random.default_rng(B)
    cand = np.stack([np.sort(rng.choice(np.arange(1, T - 2), C_cap, replace=False)) for _ in range(B)])
    cand = torch.as_tensor(cand.astype(np.int32), device=DEV)
    cnt = torch.full((B,), C_cap, dtype=torch.int32, device=DEV)
    cnt[0] = 0                                                   # no candidate: nothing waits
    L = torch.full((B,), T, dtype=torch.int32, device=DEV)
    best = torch.full((B,), 7, dtype=torch.int32, device=DEV)
    bscore = torch.zeros(B, dtype=torch.float32, device=DEV)
    status = torch.zeros(B, dtype=torch.int32, device=DEV)
    s = torch.cuda.current_stream().cuda_stream
    rc = stuck.pldp_rank_hidden(H.data_ptr(), 1, d, T * d, L.data_ptr(), B, T, cand.data_ptr(), cnt.data_ptr(),
                                C_cap, float("-inf"), None, best.data_ptr(), bscore.data_ptr(), status.data_ptr(), s)
    assert rc == 0
    torch.cuda.synchronize()                                     # the call returned and completed
    st = status.cpu().numpy()
    assert st[0] == 0 and (st[1:] == lib.PLDP_ST_TIMEOUT).all(), st
    assert best.cpu().tolist() == [-1] * B
    assert bool(torch.isneginf(bscore).all())
    # the context is still usable, and the product build takes the same inputs normally
    lib.pldp_rank_hidden(H, L, cand, cnt, best, best_score=bscore, status=status.zero_())
    torch.cuda.synchronize()
    assert (status.cpu().numpy() == 0).all() and (best.cpu().numpy()[1:] >= 1).all()
