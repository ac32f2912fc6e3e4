"""aal_accept_reward_noalloc against aal_accept_reward (GPU, through the C ABI).

The no-allocation entry point serves callers that cannot allocate device memory for a
workspace (their device memory is reserved up front by their own allocator, or they only
hold pointers handed to them).  It must give the same results as the workspace entry
point, call after call, although every call reuses the same fixed scratch array.  This
file is collected last so that a failure here comes after every other test has run.
"""

import ctypes

import numpy as np
import pytest
import torch

import paper_2609_24150_gb300 as aal
import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _outputs(N, wpr):
    return (torch.full((N,), -1, dtype=torch.int32, device=DEV),
            torch.full((N,), -1, dtype=torch.int32, device=DEV),
            torch.full((N // wpr,), float("nan"), device=DEV),
            torch.full((N // wpr,), float("nan"), device=DEV))


def _both(target, draft, ref, mode, T, seed, row_offset, wpr, rpg):
    prob = aal.reward_problem(draft, mode, T, 3.0, seed, row_offset, wpr, rpg)
    N = draft.shape[0]
    ws = torch.empty(aal.aal_reward_workspace_size(prob), dtype=torch.uint8, device=DEV)
    a = _outputs(N, wpr)
    aal.aal_accept_reward(prob, draft, target, ref, ws, a[0], a[1] if ref is not None else None, a[2], a[3])
    b = _outputs(N, wpr)
    aal.aal_accept_reward_noalloc(prob, draft, target, ref, b[0], b[1] if ref is not None else None, b[2], b[3])
    torch.cuda.synchronize()
    return [x.cpu().numpy() for x in a], [x.cpu().numpy() for x in b]


def _same(a, b, with_ref):
    np.testing.assert_array_equal(a[0], b[0])                     # tau: bit-exact
    if with_ref:
        np.testing.assert_array_equal(a[1], b[1])
    np.testing.assert_allclose(b[2], a[2], rtol=0, atol=1e-6)     # rollout lengths
    np.testing.assert_allclose(b[3], a[3], rtol=0, atol=1e-5)     # advantages


def test_noalloc_matches_workspace_entry_point_on_two_calls_in_a_row():
    # call 1: greedy with a reference draft, bf16, 64 windows of K = 8
    t1, d1, r1 = synth.make_reward_logits(0, seed=3, device=DEV, with_ref=True, windows_per_rollout=4,
                                          rollouts_per_group=16, K=8, V=5000)
    d1[::4] = t1[::4]
    a, b = _both(t1, d1, r1, aal.AAL_GREEDY, 1.0, 0, 0, 4, 4)
    _same(a, b, True)
    assert b[0].max() == 8
    # call 2: a different, smaller sampling problem without a reference draft; stale
    # contents of the shared scratch from call 1 must not leak into it
    t2, d2, _ = synth.make_reward_logits(1, seed=4, device=DEV, windows_per_rollout=2,
                                         rollouts_per_group=6, K=5, V=777, dtype=torch.float32)
    a, b = _both(t2, d2, None, aal.AAL_SAMPLING, 0.8, 99, 12345, 2, 3)
    _same(a, b, False)


def test_noalloc_rejects_problems_beyond_its_scratch():
    d = torch.empty(1, 1, 8, dtype=torch.bfloat16, device=DEV)
    prob = aal.AalRewardProblem(aal.AAL_NOALLOC_MAX_ROWS + 1, 1, 8, aal.AAL_BF16, aal.AAL_GREEDY, 1.0, 5.0,
                                0, 0, 1, 1)
    code = aal.library().aal_accept_reward_noalloc(ctypes.byref(prob), d.data_ptr(), d.data_ptr(), None,
                                                   d.data_ptr(), None, d.data_ptr(), d.data_ptr(), None)
    assert code == aal.AAL_ERR_UNSUPPORTED
