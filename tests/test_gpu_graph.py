"""The step as a CUDA graph: aal_loss_fwd, aal_loss_bwd and aal_accept_reward_from_loss launch
only kernels and async memsets on the caller's stream, so they can be captured once and replayed
(for callers with many small batches, where launch latency matters).  Replays must reproduce
eager launches bit for bit (every reduction has a fixed order)."""

import pytest
import torch

import paper_2609_24150_gb300 as aal
import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(autouse=True, scope="module")
def _fuse_short_rows():
    """The fused kernels on every row they take, short rows included (the default sends rows
    shorter than 128 KB to the two calls, which are faster there); restored afterwards."""
    aal.aal_debug_fused_min_row_bytes(0)
    yield
    aal.aal_debug_fused_min_row_bytes(-1)


@pytest.mark.parametrize("mode,T", [(aal.AAL_BOTH, 1.0), (aal.AAL_KL | aal.AAL_GREEDY, 1.0), (aal.AAL_SAMPLING, 0.8)])
def test_step_replays_bit_exactly(mode, T):
    target, draft, mask = synth.make_logits("v32k", seed=6, n_windows=256)
    t, d, m = target.to(DEV), draft.to(DEV), mask.to(DEV)
    N = d.shape[0]
    prob = aal.loss_problem(d, mode, T, 0.4, 0.6, 1.0)
    rprob = aal.reward_problem(d, aal.AAL_GREEDY, windows_per_rollout=16, rollouts_per_group=16)
    ws = torch.empty(aal.aal_workspace_size(prob), dtype=torch.uint8, device=DEV)
    rws = torch.empty(aal.aal_reward_workspace_size(rprob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    eal = torch.empty(N, 2, device=DEV)
    grad = torch.empty_like(d)
    tau = torch.empty(N, dtype=torch.int32, device=DEV)
    rl = torch.empty(N // 16, device=DEV)
    adv = torch.empty(N // 16, device=DEV)

    def step():
        aal.aal_loss_fwd(prob, d, t, m, ws, loss, eal)
        aal.aal_loss_bwd(prob, d, t, m, ws, 2.0, grad)
        aal.aal_accept_reward_from_loss(rprob, prob, ws, rws, tau, rl, adv)

    step()
    torch.cuda.synchronize()
    ref = [x.clone() for x in (loss, eal, grad, tau, adv)]
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):          # warm the launchers on the capture stream
        step()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step()
    for x in (loss, eal, grad):
        x.fill_(float("nan"))
    tau.fill_(-1)
    for _ in range(2):
        g.replay()
        torch.cuda.synchronize()
        assert aal.aal_check_device_status(ws) == aal.AAL_OK
        for a, b in zip((loss, eal, grad, tau, adv), ref):
            assert torch.equal(a, b)


@pytest.mark.parametrize("mode,T", [(aal.AAL_BOTH, 1.0), (aal.AAL_KL | aal.AAL_GREEDY, 1.0)])
def test_fused_step_replays_bit_exactly(mode, T):
    """aal_loss_fwd_bwd (async memsets, a counting kernel, the cooperative fused launch and the
    window kernel) and the reward, captured once: replays equal eager calls bit for bit."""
    target, draft, mask = synth.make_logits("v32k", seed=7, n_windows=256)
    t, d, m = target.to(DEV), draft.to(DEV), mask.to(DEV)
    N = d.shape[0]
    prob = aal.loss_problem(d, mode, T, 0.4, 0.6, 1.0)
    rprob = aal.reward_problem(d, aal.AAL_GREEDY, windows_per_rollout=16, rollouts_per_group=16)
    ws = torch.empty(aal.aal_workspace_size(prob), dtype=torch.uint8, device=DEV)
    rws = torch.empty(aal.aal_reward_workspace_size(rprob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    eal = torch.empty(N, 2, device=DEV)
    grad = torch.empty_like(d)
    tau = torch.empty(N, dtype=torch.int32, device=DEV)
    rl = torch.empty(N // 16, device=DEV)
    adv = torch.empty(N // 16, device=DEV)

    def step():
        aal.aal_loss_fwd_bwd(prob, d, t, m, ws, 2.0, loss, grad, eal)
        aal.aal_accept_reward_from_loss(rprob, prob, ws, rws, tau, rl, adv)

    step()
    torch.cuda.synchronize()
    ref = [x.clone() for x in (loss, eal, grad, tau, adv)]
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        step()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step()
    for x in (loss, eal, grad):
        x.fill_(float("nan"))
    tau.fill_(-1)
    for _ in range(2):
        g.replay()
        torch.cuda.synchronize()
        assert aal.aal_check_device_status(ws) == aal.AAL_OK
        for a, b in zip((loss, eal, grad, tau, adv), ref):
            assert torch.equal(a, b)


@pytest.mark.parametrize("masked", [False, True])
def test_fused_sequence_step_replays_bit_exactly(masked):
    """aal_seq_loss_fwd_bwd (async memsets, the count kernel, the cooperative fused launch, the
    sequence window and gather kernels) captured once: replays equal eager calls bit for bit."""
    target, draft, mask = synth.make_seq_logits("seq_tiny", seed=8, B=3, seq_len=120, V=4104,
                                                dtype=torch.bfloat16, masked=masked)
    t, d = target.to(DEV), draft.to(DEV)
    m = None if mask is None else mask.to(DEV)
    R = d.shape[0] * d.shape[1]
    prob = aal.seq_problem(d, 6, aal.AAL_BOTH, 1.0, 0.4, 0.6)
    ws = torch.empty(aal.aal_seq_workspace_size(prob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    eal = torch.empty(R, 2, device=DEV)
    grad = torch.empty_like(d)

    def step():
        aal.aal_seq_loss_fwd_bwd(prob, d, t, m, ws, 2.0, loss, grad, eal)

    step()
    torch.cuda.synchronize()
    ref = [x.clone() for x in (loss, eal, grad)]
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        step()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step()
    for x in (loss, eal, grad):
        x.fill_(float("nan"))
    for _ in range(2):
        g.replay()
        torch.cuda.synchronize()
        assert aal.aal_check_device_status(ws) == aal.AAL_OK
        for a, b in zip((loss, eal, grad), ref):
            assert torch.equal(a, b)
