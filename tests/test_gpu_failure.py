"""Failure detection on the GPU without a fault: a bounded device wait is made to run out
(a ring copy whose barrier nothing completes), the kernel reports AAL_ERR_TIMEOUT through the
workspace status word and returns, and the context stays usable for the next call."""

import pytest
import torch

import paper_2609_24150_gb300 as aal
import synth
from tests.parity import LossRun, check_loss

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


# 32 rows of V = 20000 bf16 (two ring chunks per pass), fewer rows than CTAs: each CTA
# streams one row, chunks 0-1 in the first pass and 2-3 in the second (two-pass modes only)
@pytest.mark.parametrize("mode,chunk", [(aal.AAL_BOTH, 0), (aal.AAL_BOTH, 1), (aal.AAL_BOTH, 3),
                                        (aal.AAL_KL | aal.AAL_GREEDY, 0), (aal.AAL_KL | aal.AAL_GREEDY, 1)])
def test_bounded_wait_times_out_and_context_stays_usable(mode, chunk):
    target, draft, _ = synth.make_logits("tiny", seed=11, N=16, K=2, V=20000, dtype=torch.bfloat16)
    t, d = target.to(DEV), draft.to(DEV)
    prob = aal.loss_problem(d, mode, 1.0, 0.5, 0.5)
    ws = torch.empty(aal.aal_workspace_size(prob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    aal.aal_debug_fail_next_forward(chunk, 50_000_000)        # waits give up after 50 ms
    try:
        aal.aal_loss_fwd(prob, d, t, None, ws, loss)
        assert aal.aal_check_device_status(ws) == aal.AAL_ERR_TIMEOUT
        assert aal.aal_check_device_status(ws) == aal.AAL_OK  # the status word was cleared
    finally:
        aal.aal_debug_fail_next_forward(-1, 0)                # default limit again
    # the same context runs the next forward and backward correctly
    run = LossRun(t, d, None, mode, 1.0, 0.5, 0.5, dloss=32.0)
    check_loss(run, t, d, None, mode, 1.0, 0.5, 0.5, dloss=32.0)


def test_one_tensor_stream_times_out_and_context_stays_usable():
    """The single-tensor ring (loss forward with token ids, GRPO reference pass)."""
    target, draft, _ = synth.make_logits("tiny", seed=12, N=16, K=2, V=40000, dtype=torch.bfloat16)
    t, d = target.to(DEV), draft.to(DEV)
    ids = t.float().argmax(-1).to(torch.int32).contiguous()
    mode = aal.AAL_GREEDY | aal.AAL_GRPO | aal.AAL_IDS
    prob = aal.loss_problem(d, mode, 1.0, 1.0, 0.0)
    ws = torch.empty(aal.aal_workspace_size(prob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    # 32 rows, fewer than CTAs: each CTA streams one row in two 48 KB chunks
    aal.aal_debug_fail_next_forward(1, 50_000_000)
    try:
        aal.aal_loss_fwd(prob, d, ids, None, ws, loss)
        assert aal.aal_check_device_status(ws) == aal.AAL_ERR_TIMEOUT
        assert aal.aal_check_device_status(ws) == aal.AAL_OK
        aal.aal_loss_fwd(prob, d, ids, None, ws, loss)          # clean forward
        gprob = aal.grpo_problem(d, 1, 16)
        gws = torch.empty(aal.aal_grpo_workspace_size(gprob), dtype=torch.uint8, device=DEV)
        gl = torch.empty(1, device=DEV)
        aal.aal_debug_fail_next_forward(0, 50_000_000)
        aal.aal_grpo_from_loss(gprob, prob, ws, d, gws, gl)
        assert aal.aal_check_device_status(gws) == aal.AAL_ERR_TIMEOUT
        assert aal.aal_check_device_status(gws) == aal.AAL_OK
    finally:
        aal.aal_debug_fail_next_forward(-1, 0)
    # the same context still computes the right greedy loss from ids
    run = LossRun(ids, d, None, aal.AAL_GREEDY | aal.AAL_IDS, 1.0, 1.0, 0.0, dloss=32.0)
    check_loss(run, t, d, None, aal.AAL_GREEDY, 1.0, 1.0, 0.0, dloss=32.0)
