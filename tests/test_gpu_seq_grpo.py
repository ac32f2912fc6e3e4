"""GPU parity of the GRPO stage over sequences (aal_seq_grpo_from_loss, Sec. 3.4): the window
samples are sliced from one forward pass per sequence, groups of m consecutive windows at a few
anchors, and each position's gradient adds every window that covers it."""

import numpy as np
import pytest
import torch

import oracle
import paper_2609_24150_gb300 as aal
import synth
from oracle.sequence import seq_grpo_backward, seq_grpo_forward, slice_windows
from tests.parity import GRAD_ATOL, GRAD_RTOL, LOSS_ATOL, LOSS_RTOL
from tests.test_gpu_grpo import _near_edges

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
MODE = aal.AAL_KL | aal.AAL_GREEDY | aal.AAL_GRPO


def _starts(anchors_per_seq, m, T):
    """Groups of m consecutive windows at each anchor, flat and ascending."""
    out = []
    for b, anchors in enumerate(anchors_per_seq):
        for a in sorted(anchors):
            out += [b * T + a + i for i in range(m)]
    return torch.tensor(sorted(out), dtype=torch.int32)


class SeqGrpoStep:
    def __init__(self, target, draft, ref, mask, starts, K, m, dloss, wg=0.1, wkl=1.0, w_grpo=0.1, eps=0.2):
        B, T, V = draft.shape
        N = starts.numel()
        self.sprob = aal.seq_problem(draft, K, MODE, 1.0, wg, 0.0, False, wkl)
        self.lws = torch.empty(aal.aal_seq_workspace_size(self.sprob), dtype=torch.uint8, device=DEV)
        self.loss = torch.empty(1, device=DEV)
        aal.aal_seq_loss_fwd(self.sprob, draft, target, mask, self.lws, self.loss)
        self.gprob = aal.grpo_seq_problem(N, draft, K, 1, m, eps_clip=eps, w_grpo=w_grpo)
        self.gws = torch.empty(aal.aal_seq_grpo_workspace_size(self.gprob, self.sprob), dtype=torch.uint8,
                               device=DEV)
        self.gloss = torch.empty(1, device=DEV)
        self.tau = torch.empty(N, dtype=torch.int32, device=DEV)
        self.tau_ref = torch.empty(N, dtype=torch.int32, device=DEV)
        self.adv = torch.empty(N, device=DEV)
        self.log_rho = torch.empty(N, device=DEV)
        aal.aal_seq_grpo_from_loss(self.gprob, self.sprob, self.lws, ref, starts.to(DEV), self.gws, self.gloss,
                                   self.tau, self.tau_ref, self.adv, self.log_rho)
        self.grad = torch.empty_like(draft)
        aal.aal_seq_loss_bwd(self.sprob, draft, target, mask, self.lws, dloss, self.grad)
        torch.cuda.synchronize()
        self.status = aal.aal_check_device_status(self.gws)
        assert aal.aal_check_device_status(self.lws) == aal.AAL_OK


@pytest.mark.parametrize("V,dtype", [(1000, torch.float32), (4104, torch.bfloat16), (7, torch.bfloat16)])
def test_small_sequences_every_position(V, dtype):
    B, T, K, m = 2, 24, 3, 4
    target, draft, mask = synth.make_seq_logits("seq_tiny", seed=V, B=B, seq_len=T, V=V, dtype=dtype)
    g = torch.Generator().manual_seed(V)
    ref = (draft.float() + 0.3 * torch.randn(draft.shape, generator=g)).to(dtype)
    draft[:, ::2] = target[:, ::2]                  # positions that the greedy draft gets right
    starts = _starts([[0, 9], [2, 14]], m, T)
    t, d, r, msk = [x.to(DEV) for x in (target, draft, ref, mask)]
    dloss = 48.0
    step = SeqGrpoStep(t, d, r, msk, starts, K, m, dloss)
    assert step.status == aal.AAL_OK
    st = starts.numpy()
    kw = dict(windows_per_rollout=1, rollouts_per_group=m, adv_clip=5.0, eps_clip=0.2, rho_min=0.0,
              rho_max=10.0, log_rho_clip=10.0)
    fw = seq_grpo_forward(target, draft, ref, st, K, **kw)
    np.testing.assert_array_equal(step.tau.cpu().numpy(), fw["reward"]["tau"])
    np.testing.assert_array_equal(step.tau_ref.cpu().numpy(), fw["reward"]["tau_ref"])
    np.testing.assert_allclose(step.adv.cpu().numpy(), fw["reward"]["advantage"], rtol=1e-6, atol=1e-6)
    np.testing.assert_allclose(step.log_rho.cpu().numpy(), fw["log_rho"], rtol=1e-5, atol=2e-5)
    assert abs(step.gloss.item() - fw["loss"]) <= LOSS_RTOL * abs(fw["loss"]) + 1e-5
    m_h = mask.numpy()
    omode = oracle.MODE_KL | oracle.MODE_GREEDY
    ref_loss = oracle.seq_objective_forward(target, draft, m_h, K, omode, 1.0, 0.1, 0.0, 1.0)["loss"]
    assert abs(step.loss.item() - ref_loss) <= LOSS_RTOL * abs(ref_loss) + LOSS_ATOL
    g_ref = oracle.seq_objective_backward(target, draft, m_h, K, omode, 1.0, 0.1, 0.0, 1.0, dloss)
    g_ref = g_ref + seq_grpo_backward(target, draft, ref, st, K, dloss=dloss * 0.1, **kw)
    # positions covered by a window whose ratio sits on a clip edge are set aside
    near = _near_edges(fw, kw)
    keep = np.ones((B * T,), dtype=bool)
    for n in np.flatnonzero(near):
        keep[st[n]:st[n] + K] = False
    keep = keep.reshape(B, T)
    gg = step.grad.double().cpu().numpy()
    bad = (np.abs(gg - g_ref) > GRAD_ATOL + GRAD_RTOL * np.abs(g_ref)) & keep[..., None]
    assert not bad.any(), (int(bad.sum()), tuple(np.argwhere(bad)[0]))


def test_unsorted_or_outside_starts_are_reported():
    B, T, K, V = 1, 20, 3, 1000
    target, draft, _ = synth.make_seq_logits("seq_tiny", seed=5, B=B, seq_len=T, V=V, masked=False)
    t, d = target.to(DEV), draft.to(DEV)
    for bad in ([5, 3, 7, 8], [0, 1, 2, 18]):      # descending; crossing the sequence end
        step = SeqGrpoStep(t, d, d.clone(), None, torch.tensor(bad, dtype=torch.int32), K, 4, 4.0)
        assert step.status == aal.AAL_ERR_INVALID_ARG
        assert torch.isfinite(step.grad).all()


def test_full_size_sampled_windows_and_positions():
    """seq_v128k (4 x 2048 positions, K = 7, V = 128256 bf16), 8 anchors per sequence with groups of
    16 windows: tau, tau^ref and log rho of sampled windows against the oracle, the advantages as the
    oracle standardises the GPU's rewards, the loss as the mean of the windows' surrogates, and the
    GRPO part of sampled positions' gradient rows (the forward's own terms are checked elsewhere:
    here the step without the GRPO call is subtracted)."""
    target, draft, mask = synth.make_seq_logits("seq_v128k", seed=3, device=DEV)
    B, T, V = draft.shape
    K, m = 7, 16
    g = torch.Generator(device=DEV).manual_seed(3)
    ref = (draft.float() + 0.3 * torch.randn(draft.shape, generator=g, device=DEV)).to(draft.dtype)
    valid = mask.cpu().numpy()
    anchors = []
    for b in range(B):
        v = np.flatnonzero(valid[b])
        lo, hi = int(v[0]), int(v[-1]) - K - m
        anchors.append(list(np.linspace(lo, hi, 8).astype(int) // (m + 1) * (m + 1)))
    starts = _starts(anchors, m, T)
    N = starts.numel()
    dloss = float(N)
    step = SeqGrpoStep(target, draft, ref, mask, starts, K, m, dloss, w_grpo=1.0)
    assert step.status == aal.AAL_OK
    # the same forward and backward without the GRPO term
    base = torch.empty_like(draft)
    sprob0 = aal.seq_problem(draft, K, aal.AAL_KL | aal.AAL_GREEDY, 1.0, 0.1, 0.0, False, 1.0)
    lws0 = torch.empty(aal.aal_seq_workspace_size(sprob0), dtype=torch.uint8, device=DEV)
    l0 = torch.empty(1, device=DEV)
    aal.aal_seq_loss_fwd(sprob0, draft, target, mask, lws0, l0)
    aal.aal_seq_loss_bwd(sprob0, draft, target, mask, lws0, dloss, base)
    torch.cuda.synchronize()
    st = starts.numpy()
    tau, tau_ref, adv, lr = (x.cpu().numpy() for x in (step.tau, step.tau_ref, step.adv, step.log_rho))
    R = tau.astype(np.float64) - tau_ref
    np.testing.assert_allclose(adv, oracle.group_advantages(oracle.rollout_lengths(R, 1), m, 5.0), atol=1e-6)
    rho = np.clip(np.exp(lr), 0.0, 10.0)
    surr = np.minimum(rho * adv, np.clip(rho, 0.8, 1.2) * adv)
    assert abs(step.gloss.item() + surr.sum() / N) <= 1e-4 * abs(surr.sum() / N) + 1e-6
    kw = dict(windows_per_rollout=1, rollouts_per_group=m, adv_clip=5.0, eps_clip=0.2, rho_min=0.0,
              rho_max=10.0, log_rho_clip=10.0)
    sel = [0, 5, N // 2, N - 1]
    sub = st[sel]
    fw = seq_grpo_forward(target.cpu(), draft.cpu(), ref.cpu(), sub, K, advantage_window=adv[sel].astype(np.float64),
                          n_windows_total=N, **kw)
    np.testing.assert_allclose(lr[sel], fw["log_rho"], rtol=1e-5, atol=2e-5)
    rw = oracle.accept_reward(slice_windows(target.cpu(), sub, K), slice_windows(draft.cpu(), sub, K),
                              slice_windows(ref.cpu(), sub, K), 1)
    np.testing.assert_array_equal(tau[sel], rw["tau"])
    np.testing.assert_array_equal(tau_ref[sel], rw["tau_ref"])
    # GRPO part of the gradient at positions covered by a few windows
    grpo_part = (step.grad.float() - base.float())
    for p in [int(st[0]) + 2, int(st[N // 2]) + K - 1]:
        cover = [n for n in range(N) if st[n] <= p < st[n] + K]
        want = np.zeros(V)
        for n in cover:
            gw = oracle.grpo_backward(slice_windows(target.cpu(), [st[n]], K), slice_windows(draft.cpu(), [st[n]], K),
                                      slice_windows(ref.cpu(), [st[n]], K), dloss=dloss,
                                      advantage_window=adv[[n]].astype(np.float64), n_windows_total=N, **kw)
            want += gw[0, p - st[n]]
        got = grpo_part.view(B * T, V)[p].double().cpu().numpy()
        assert np.all(np.abs(got - want) <= 4e-5 + 2e-2 * np.abs(want)), (p, np.abs(got - want).max())
