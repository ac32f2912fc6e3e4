"""GPU parity of target token-id input (mode bit AAL_IDS): x* given as int32 ids, only the
draft read (Sec. 3.2: for greedy target-generated data x* is the ground-truth token)."""

import numpy as np
import pytest
import torch

import oracle
import paper_2609_24150_gb300 as aal
import synth
from tests.parity import GRAD_ATOL, GRAD_RTOL, LOSS_ATOL, LOSS_RTOL, LossRun, SeqRun

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
G_IDS = aal.AAL_GREEDY | aal.AAL_IDS


def _dev(*ts):
    return [None if t is None else t.to(DEV) for t in ts]


def _ids_of(target):
    return target.float().argmax(-1).to(torch.int32).contiguous()


def _check_windowed(run, draft, ids, mask, wg, dloss):
    d_h = draft.cpu()
    ids_h = ids.cpu().numpy()
    m_h = None if mask is None else mask.cpu().numpy()
    fw = oracle.loss_forward(None, d_h, m_h, oracle.MODE_GREEDY, 1.0, wg, 0.0, xstar=ids_h)
    np.testing.assert_allclose(run.eal.cpu().numpy()[:, 0], fw["eal_g"], rtol=LOSS_RTOL, atol=LOSS_ATOL)
    assert abs(run.loss.item() - fw["loss"]) <= LOSS_RTOL * abs(fw["loss"]) + LOSS_ATOL
    g_ref = oracle.loss_backward(None, d_h, m_h, oracle.MODE_GREEDY, 1.0, wg, 0.0, dloss, xstar=ids_h)
    g = run.grad.double().cpu().numpy()
    bad = np.abs(g - g_ref) > GRAD_ATOL + GRAD_RTOL * np.abs(g_ref)
    assert not bad.any(), (int(bad.sum()), tuple(np.argwhere(bad)[0]))


@pytest.mark.parametrize("V,dtype", [(1000, torch.float32), (4104, torch.bfloat16), (7, torch.bfloat16),
                                     (4099, torch.float32), (65544, torch.bfloat16)])
@pytest.mark.parametrize("K", [1, 4])
def test_ids_all_rows(V, dtype, K):
    """Streamed (16-byte rows) and plain (other rows) one-tensor passes; ids drawn uniformly, so
    x* is usually not the draft's argmax."""
    _, draft, _ = synth.make_logits("tiny", seed=V + K, N=12, K=K, V=V, dtype=dtype)
    g = torch.Generator().manual_seed(V)
    ids = torch.randint(0, V, (12, K), generator=g, dtype=torch.int32)
    mask = torch.ones(12, K, dtype=torch.uint8)
    mask[3, 0] = 0
    if K > 1:
        mask[5, 2] = 0
    d, i, m = _dev(draft, ids, mask)
    dloss = 12.0 * K
    run = LossRun(i, d, m, G_IDS, 1.0, 0.7, 0.0, dloss=dloss)
    _check_windowed(run, d, i, m, 0.7, dloss)


def test_ids_match_the_target_logit_path():
    """ids = argmax of the target logits: the same expected lengths and gradient as the
    forward that reads the target (to fp32 rounding), and the same draft tokens (the greedy
    reward from the statistics is bit-identical)."""
    target, draft, _ = synth.make_logits("v32k", seed=4, n_windows=256)
    t, d = _dev(target, draft)
    ids = _ids_of(t)
    a = LossRun(ids, d, None, G_IDS, 1.0, 1.0, 0.0, dloss=256.0 * 5)
    b = LossRun(t, d, None, aal.AAL_GREEDY, 1.0, 1.0, 0.0, dloss=256.0 * 5)
    np.testing.assert_allclose(a.eal.cpu().numpy(), b.eal.cpu().numpy(), rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(a.grad.float().cpu().numpy(), b.grad.float().cpu().numpy(), rtol=2e-2, atol=2e-5)
    taus = []
    for run in (a, b):
        rprob = aal.reward_problem(d, aal.AAL_GREEDY, windows_per_rollout=16, rollouts_per_group=16)
        rws = torch.empty(aal.aal_reward_workspace_size(rprob), dtype=torch.uint8, device=DEV)
        tau = torch.empty(256, dtype=torch.int32, device=DEV)
        rl = torch.empty(16, device=DEV)
        adv = torch.empty(16, device=DEV)
        aal.aal_accept_reward_from_loss(rprob, run.prob, run.ws_buf, rws, tau, rl, adv)
        taus.append(tau.cpu())
    assert torch.equal(taus[0], taus[1])


def test_out_of_range_ids_are_reported():
    _, draft, _ = synth.make_logits("tiny", seed=2, N=4, K=3, V=4104, dtype=torch.bfloat16)
    d = draft.to(DEV)
    ids = torch.zeros(4, 3, dtype=torch.int32, device=DEV)
    ids[1, 2] = 4104          # one past the end
    ids[2, 0] = -5
    prob = aal.loss_problem(d, G_IDS, 1.0, 1.0, 0.0)
    ws = torch.empty(aal.aal_workspace_size(prob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    eal = torch.empty(4, 2, device=DEV)
    aal.aal_loss_fwd(prob, d, ids, None, ws, loss, eal)
    assert aal.aal_check_device_status(ws) == aal.AAL_ERR_INVALID_ARG
    assert aal.aal_check_device_status(ws) == aal.AAL_OK
    e = eal[:, 0].cpu()
    assert e[2].item() == 0.0              # a^g = 0 at depth 0 ends the window
    assert torch.isfinite(loss).all()


@pytest.mark.parametrize("V,dtype", [(1000, torch.float32), (4104, torch.bfloat16), (7, torch.bfloat16)])
def test_ids_sequence_layout(V, dtype):
    target, draft, mask = synth.make_seq_logits("seq_tiny", seed=V, V=V, dtype=dtype)
    t, d, m = _dev(target, draft, mask)
    ids = _ids_of(t)
    K = 4
    dloss = float(m.sum().item())
    run = SeqRun(ids, d, m, K, G_IDS, 1.0, 1.0, 0.0, dloss=dloss)
    ids_h = ids.cpu().numpy()
    fw = oracle.seq_loss_forward(None, d.cpu(), m.cpu().numpy(), K, oracle.MODE_GREEDY, xstar=ids_h)
    np.testing.assert_allclose(run.eal.cpu().numpy()[:, 0], fw["eal_g"], rtol=LOSS_RTOL, atol=LOSS_ATOL)
    assert abs(run.loss.item() - fw["loss"]) <= LOSS_RTOL * abs(fw["loss"]) + LOSS_ATOL
    g_ref = oracle.seq_loss_backward(None, d.cpu(), m.cpu().numpy(), K, oracle.MODE_GREEDY, dloss=dloss, xstar=ids_h)
    g = run.grad.double().cpu().numpy()
    assert not (np.abs(g - g_ref) > GRAD_ATOL + GRAD_RTOL * np.abs(g_ref)).any()


def test_grpo_step_on_ids():
    """L_EAL + 0.1 L_GRPO with x* as ids: tau^theta and tau^ref against the oracle with a target
    peaked on the ids, and the loss and gradient as the logit path gives them."""
    parts = [synth.make_reward_logits(g, seed=12, with_ref=True, windows_per_rollout=1, rollouts_per_group=8, K=3,
                                      V=4104, dtype=torch.bfloat16, ref_from_draft=0.3) for g in range(2)]
    t, d, r = [torch.cat([p[i] for p in parts]).to(DEV) for i in range(3)]
    ids = _ids_of(t)
    out = []
    for mode, tgt in [(aal.AAL_GREEDY | aal.AAL_GRPO | aal.AAL_IDS, ids), (aal.AAL_GREEDY | aal.AAL_GRPO, t)]:
        lprob = aal.loss_problem(d, mode, 1.0, 1.0, 0.0)
        lws = torch.empty(aal.aal_workspace_size(lprob), dtype=torch.uint8, device=DEV)
        loss = torch.empty(1, device=DEV)
        aal.aal_loss_fwd(lprob, d, tgt, None, lws, loss)
        gprob = aal.grpo_problem(d, 1, 8, w_grpo=0.1)
        gws = torch.empty(aal.aal_grpo_workspace_size(gprob), dtype=torch.uint8, device=DEV)
        gl = torch.empty(1, device=DEV)
        tau = torch.empty(16, dtype=torch.int32, device=DEV)
        tau_ref = torch.empty(16, dtype=torch.int32, device=DEV)
        aal.aal_grpo_from_loss(gprob, lprob, lws, r, gws, gl, tau, tau_ref)
        grad = torch.empty_like(d)
        aal.aal_loss_bwd(lprob, d, tgt, None, lws, 48.0, grad)
        torch.cuda.synchronize()
        assert aal.aal_check_device_status(lws) == aal.AAL_OK
        out.append((loss.item(), gl.item(), tau.cpu(), tau_ref.cpu(), grad.float().cpu()))
    rw = oracle.accept_reward(t.cpu(), d.cpu(), r.cpu(), 1, windows_per_rollout=1, rollouts_per_group=8)
    assert np.array_equal(out[0][2].numpy(), rw["tau"]) and np.array_equal(out[0][3].numpy(), rw["tau_ref"])
    assert torch.equal(out[0][2], out[1][2]) and torch.equal(out[0][3], out[1][3])
    assert abs(out[0][0] - out[1][0]) <= 1e-5 * abs(out[1][0]) + 1e-6
    assert abs(out[0][1] - out[1][1]) <= 1e-5 * abs(out[1][1]) + 1e-6
    np.testing.assert_allclose(out[0][4].numpy(), out[1][4].numpy(), rtol=2e-2, atol=2e-5)


def test_full_size_ids_match_the_logit_path():
    """v128k (8192 windows x K = 7, V = 128256 bf16) with ids = argmax z_p: the draft's greedy
    tokens give bit-identical greedy rewards, the expected lengths agree to fp32 rounding, and
    sampled windows match the oracle."""
    target, draft, _ = synth.make_logits("v128k", seed=1, device=DEV)
    ids = _ids_of(target)
    N, K, V = draft.shape
    a = LossRun(ids, draft, None, G_IDS, 1.0, 1.0, 0.0, dloss=float(N * K))
    eal_ids, grad_rows = a.eal.clone(), a.grad[[0, 4000, 8191]].clone()
    taus = []
    for tgt, mode in [(ids, G_IDS), (target, aal.AAL_GREEDY)]:
        run = a if mode == G_IDS else LossRun(tgt, draft, None, mode, 1.0, 1.0, 0.0, dloss=float(N * K))
        rprob = aal.reward_problem(draft, aal.AAL_GREEDY, windows_per_rollout=256, rollouts_per_group=16)
        rws = torch.empty(aal.aal_reward_workspace_size(rprob), dtype=torch.uint8, device=DEV)
        tau = torch.empty(N, dtype=torch.int32, device=DEV)
        rl = torch.empty(N // 256, device=DEV)
        adv = torch.empty(N // 256, device=DEV)
        aal.aal_accept_reward_from_loss(rprob, run.prob, run.ws_buf, rws, tau, rl, adv)
        taus.append(tau.cpu())
        if mode == aal.AAL_GREEDY:
            np.testing.assert_allclose(eal_ids.cpu().numpy(), run.eal.cpu().numpy(), rtol=1e-5, atol=1e-6)
    assert torch.equal(taus[0], taus[1])
    sel = [0, 4000, 8191]
    d_h = draft[sel].cpu()
    ids_h = ids[sel].cpu().numpy()
    fw = oracle.loss_forward(None, d_h, None, oracle.MODE_GREEDY, 1.0, 1.0, 0.0, n_windows_total=N, xstar=ids_h)
    np.testing.assert_allclose(eal_ids.cpu().numpy()[sel, 0], fw["eal_g"], rtol=LOSS_RTOL, atol=LOSS_ATOL)
    g_ref = oracle.loss_backward(None, d_h, None, oracle.MODE_GREEDY, 1.0, 1.0, 0.0, float(N * K),
                                 n_windows_total=N, xstar=ids_h)
    g = grad_rows.double().cpu().numpy()
    assert not (np.abs(g - g_ref) > GRAD_ATOL + GRAD_RTOL * np.abs(g_ref)).any()
