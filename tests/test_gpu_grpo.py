"""GPU parity of the GRPO stage (Sec. 3.4) against the fp64 oracle, through the C ABI.

One step is aal_loss_fwd (mode with AAL_GRPO), aal_grpo_from_loss over the reference draft,
then aal_loss_bwd, whose gradient is that of the forward's objective plus w_grpo * L_GRPO.
The paper's GRPO-phase objective is L_KL + 0.1 L_EAL + 0.1 L_GRPO.
"""

import numpy as np
import pytest
import torch

import oracle
import paper_2609_24150_gb300 as aal
import synth
from tests.parity import GRAD_ATOL, GRAD_RTOL, LOSS_ATOL, LOSS_RTOL, ORACLE_MODES, grad_tolerance

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
PAPER_MODE = aal.AAL_KL | aal.AAL_GREEDY | aal.AAL_GRPO
BOUNDARY_BAND = 1e-4   # windows this close (relative) to a clip edge are decided in fp32 either way


REF_SIGMA = 0.3        # the reference policy: the draft plus N(0, 0.3^2), an earlier snapshot


def _batch(groups, wpr, rpg, K, V, dtype, seed=0):
    parts = [synth.make_reward_logits(g, seed=seed, with_ref=True, windows_per_rollout=wpr,
                                      rollouts_per_group=rpg, K=K, V=V, dtype=dtype, ref_from_draft=REF_SIGMA)
             for g in range(groups)]
    return [torch.cat([p[i] for p in parts]).to(DEV) for i in range(3)]


class GrpoStep:
    def __init__(self, target, draft, ref, lmode, T=1.0, wg=0.1, ws=0.0, wkl=1.0, dloss=1.0, call_grpo=True,
                 **gp):
        N, K, V = draft.shape
        self.lprob = aal.loss_problem(draft, lmode, T, wg, ws, wkl)
        self.lws = torch.empty(aal.aal_workspace_size(self.lprob), dtype=torch.uint8, device=DEV)
        self.loss = torch.full((1,), float("nan"), device=DEV)
        aal.aal_loss_fwd(self.lprob, draft, target, None, self.lws, self.loss)
        self.gprob = aal.grpo_problem(draft, **gp)
        self.gws = torch.empty(aal.aal_grpo_workspace_size(self.gprob), dtype=torch.uint8, device=DEV)
        self.gloss = torch.full((1,), float("nan"), device=DEV)
        nroll = N // self.gprob.windows_per_rollout
        self.tau = torch.full((N,), -1, dtype=torch.int32, device=DEV)
        self.tau_ref = torch.full((N,), -1, dtype=torch.int32, device=DEV)
        self.adv = torch.full((nroll,), float("nan"), device=DEV)
        self.log_rho = torch.full((N,), float("nan"), device=DEV)
        if call_grpo:
            aal.aal_grpo_from_loss(self.gprob, self.lprob, self.lws, ref, self.gws, self.gloss, self.tau,
                                   self.tau_ref, self.adv, self.log_rho)
        self.grad = torch.full_like(draft, float("nan"))
        aal.aal_loss_bwd(self.lprob, draft, target, None, self.lws, dloss, self.grad)
        torch.cuda.synchronize()
        assert aal.aal_check_device_status(self.lws) == aal.AAL_OK


def _gp(gp):
    """Oracle keyword arguments of a grpo_problem keyword set."""
    return dict(windows_per_rollout=gp.get("windows_per_rollout", 1),
                rollouts_per_group=gp.get("rollouts_per_group", 1), adv_clip=gp.get("adv_clip", 5.0),
                eps_clip=gp.get("eps_clip", 0.2), rho_min=gp.get("rho_min", 0.0),
                rho_max=gp.get("rho_max", 10.0), log_rho_clip=gp.get("log_rho_clip", 10.0))


def _near_edges(fw, kw):
    """Windows whose ratio sits within BOUNDARY_BAND of a clip edge (either decision is right)."""
    eps, c = kw["eps_clip"], kw["log_rho_clip"]
    near = np.zeros(fw["rho"].shape, dtype=bool)
    for val, edge in [(fw["rho"], 1 + eps), (fw["rho"], 1 - eps), (fw["rho_exp"], kw["rho_min"]),
                      (fw["rho_exp"], kw["rho_max"]), (fw["log_rho_raw"], c), (fw["log_rho_raw"], -c)]:
        near |= np.abs(val - edge) <= BOUNDARY_BAND * max(1.0, abs(edge))
    return near


def _check(step, target, draft, ref, lmode, T, wg, ws, wkl, dloss, gp, check_loss=True):
    kw = _gp(gp)
    w_grpo = gp.get("w_grpo", 1.0)
    t_h, d_h, r_h = target.cpu(), draft.cpu(), ref.cpu()
    rw = oracle.accept_reward(t_h, d_h, r_h, 1, windows_per_rollout=kw["windows_per_rollout"],
                              rollouts_per_group=kw["rollouts_per_group"], adv_clip=kw["adv_clip"])
    np.testing.assert_array_equal(step.tau.cpu().numpy(), rw["tau"])
    np.testing.assert_array_equal(step.tau_ref.cpu().numpy(), rw["tau_ref"])
    np.testing.assert_allclose(step.adv.cpu().numpy(), rw["advantage"], rtol=1e-6, atol=1e-6)
    fw = oracle.grpo_forward(t_h, d_h, r_h, **kw)
    np.testing.assert_allclose(step.log_rho.cpu().numpy(), fw["log_rho"], rtol=1e-5, atol=2e-5)
    got = step.gloss.item()
    assert abs(got - fw["loss"]) <= LOSS_RTOL * abs(fw["loss"]) + 1e-5, (got, fw["loss"])
    omode = ORACLE_MODES[lmode & 7] if lmode & 7 else 0
    fo = oracle.objective_forward(t_h, d_h, None, omode, T, wg, ws, wkl) if omode else None
    if check_loss:
        ref_loss = fo["loss"] if omode else 0.0
        assert abs(step.loss.item() - ref_loss) <= LOSS_RTOL * abs(ref_loss) + LOSS_ATOL
    g_ref = oracle.grpo_backward(t_h, d_h, r_h, **kw, dloss=dloss * w_grpo)
    if omode:
        g_ref = g_ref + oracle.objective_backward(t_h, d_h, None, omode, T, wg, ws, wkl, dloss)
    keep = ~_near_edges(fw, kw)
    g = step.grad.double().cpu().numpy()
    if omode & oracle.MODE_SAMPLING:    # WTV near-ties, widened as in every loss test
        tol = grad_tolerance(t_h, d_h, None, omode, T, wg, ws, dloss, g_ref, fo["nvalid"], fo)
    else:
        tol = GRAD_ATOL + GRAD_RTOL * np.abs(g_ref)
    bad = (np.abs(g - g_ref) > tol) & keep[:, None, None]
    assert not bad.any(), (int(bad.sum()), tuple(np.argwhere(bad)[0]))
    assert keep.sum() >= 0.9 * keep.size
    return fw


@pytest.mark.parametrize("wpr,rpg", [(1, 4), (2, 4), (4, 2)])
def test_paper_objective_tiny(wpr, rpg):
    """L_KL + 0.1 L_EAL + 0.1 L_GRPO, 4 groups, K = 4, V = 1000 fp32, every output."""
    target, draft, ref = _batch(4, wpr, rpg, 4, 1000, torch.float32, seed=3)
    N, K = draft.shape[:2]
    gp = dict(windows_per_rollout=wpr, rollouts_per_group=rpg, w_grpo=0.1)
    step = GrpoStep(target, draft, ref, PAPER_MODE, dloss=float(N * K), **gp)
    _check(step, target, draft, ref, PAPER_MODE, 1.0, 0.1, 0.0, 1.0, float(N * K), gp)


@pytest.mark.parametrize("lmode,T", [
    (aal.AAL_GRPO, 1.0),                                         # the surrogate alone
    (aal.AAL_BOTH | aal.AAL_GRPO, 1.0),                          # streamed forward, q1 = q~
    (aal.AAL_SAMPLING | aal.AAL_GRPO, 0.8),                      # streamed forward with its own q1
    (aal.AAL_KL | aal.AAL_BOTH | aal.AAL_GRPO, 1.0),
])
@pytest.mark.parametrize("V,dtype", [(4104, torch.bfloat16), (4099, torch.float32), (7, torch.bfloat16)])
def test_modes_and_row_kernels(lmode, T, V, dtype):
    target, draft, ref = _batch(2, 1, 8, 3, V, dtype, seed=V)
    N, K = draft.shape[:2]
    gp = dict(windows_per_rollout=1, rollouts_per_group=8, w_grpo=0.5, eps_clip=0.3)
    step = GrpoStep(target, draft, ref, lmode, T=T, wg=0.4, ws=0.6, wkl=1.0, dloss=float(N * K), **gp)
    _check(step, target, draft, ref, lmode, T, 0.4, 0.6, 1.0, float(N * K), gp)
    if lmode == aal.AAL_GRPO:
        assert step.loss.item() == 0.0


def test_ratio_clips_stop_the_gradient():
    target, draft, ref = _batch(2, 1, 8, 3, 1000, torch.float32, seed=5)
    N, K = draft.shape[:2]
    gp = dict(windows_per_rollout=1, rollouts_per_group=8, rho_min=0.9, rho_max=1.05, log_rho_clip=0.3,
              eps_clip=0.02)
    step = GrpoStep(target, draft, ref, aal.AAL_GRPO, dloss=float(N * K), **gp)
    fw = _check(step, target, draft, ref, aal.AAL_GRPO, 1.0, 0.0, 0.0, 0.0, float(N * K), gp)
    clipped = (fw["rho_exp"] < 0.9) | (fw["rho_exp"] > 1.05)
    assert clipped.any()
    g = step.grad.float().abs().amax(dim=(1, 2)).cpu().numpy()
    assert np.all(g[clipped & ~_near_edges(fw, _gp(gp))] == 0.0)


def test_identical_reference_gives_rho_one():
    target, draft, _ = _batch(2, 1, 8, 4, 3000, torch.bfloat16, seed=6)
    gp = dict(windows_per_rollout=1, rollouts_per_group=8, adv_clip=100.0)
    step = GrpoStep(target, draft, draft.clone(), aal.AAL_GRPO, **gp)
    assert float(step.log_rho.abs().max()) < 2e-5
    assert abs(step.gloss.item()) < 1e-5
    np.testing.assert_array_equal(step.tau.cpu().numpy(), step.tau_ref.cpu().numpy())


def test_without_the_grpo_call_the_term_is_zero():
    """aal_loss_fwd clears the coefficients: skipping aal_grpo_from_loss leaves the objective's
    own gradient (a workspace reused from a GRPO step must not leak its coefficients)."""
    target, draft, ref = _batch(1, 1, 8, 3, 1000, torch.float32, seed=7)
    gp = dict(windows_per_rollout=1, rollouts_per_group=8)
    first = GrpoStep(target, draft, ref, PAPER_MODE, **gp)
    lprob = first.lprob
    aal.aal_loss_fwd(lprob, draft, target, None, first.lws, first.loss)
    grad = torch.empty_like(draft)
    aal.aal_loss_bwd(lprob, draft, target, None, first.lws, 1.0, grad)
    base = GrpoStep(target, draft, ref, aal.AAL_KL | aal.AAL_GREEDY, call_grpo=False, **gp)
    torch.cuda.synchronize()
    assert torch.equal(grad, base.grad)


def test_full_prompt_group_sampled_windows():
    """One prompt group of the reward workload (16 rollouts x 256 windows, K = 8, V = 128256
    bf16) under L_KL + 0.1 L_EAL + 0.1 L_GRPO: tau, tau^ref, log rho and gradient rows of sampled
    windows against the oracle (given the group's advantages), the advantages against the
    oracle's standardisation of the GPU's rewards, and the loss against its windows' surrogates."""
    target, draft, ref = synth.make_reward_logits(0, seed=0, with_ref=True, device=DEV, ref_from_draft=REF_SIGMA)
    N, K, V = draft.shape
    gp = dict(windows_per_rollout=1, rollouts_per_group=16, w_grpo=0.1)   # groups of m = 16 windows
    step = GrpoStep(target, draft, ref, PAPER_MODE, dloss=float(N * K), **gp)
    tau = step.tau.cpu().numpy()
    tau_ref = step.tau_ref.cpu().numpy()
    adv = step.adv.cpu().numpy()
    R = tau.astype(np.float64) - tau_ref
    np.testing.assert_allclose(adv, oracle.group_advantages(oracle.rollout_lengths(R, 1), 16, 5.0),
                               rtol=1e-6, atol=1e-6)
    kw = _gp(gp)
    lr = step.log_rho.cpu().numpy()
    rho = np.clip(np.exp(lr), kw["rho_min"], kw["rho_max"])
    surr = np.minimum(rho * adv, np.clip(rho, 0.8, 1.2) * adv)
    assert abs(step.gloss.item() + surr.sum() / N) <= 1e-4 * abs(surr.sum() / N) + 1e-6
    sel = [0, 1, 777, 2048, N - 1]
    idx = torch.as_tensor(sel, device=DEV)
    t_h, d_h, r_h = target[idx].cpu(), draft[idx].cpu(), ref[idx].cpu()
    rw = oracle.accept_reward(t_h, d_h, r_h, 1)
    np.testing.assert_array_equal(tau[sel], rw["tau"])
    np.testing.assert_array_equal(tau_ref[sel], rw["tau_ref"])
    fw = oracle.grpo_forward(t_h, d_h, r_h, **kw, advantage_window=adv[sel].astype(np.float64),
                             n_windows_total=N)
    np.testing.assert_allclose(lr[sel], fw["log_rho"], rtol=1e-5, atol=2e-5)
    g_ref = oracle.grpo_backward(t_h, d_h, r_h, **kw, dloss=float(N * K) * 0.1,
                                 advantage_window=adv[sel].astype(np.float64), n_windows_total=N)
    g_ref = g_ref + oracle.objective_backward(t_h, d_h, None, ORACLE_MODES[aal.AAL_KL | aal.AAL_GREEDY], 1.0,
                                              0.1, 0.0, 1.0, float(N * K), n_windows_total=N,
                                              n_positions_total=N * K)
    keep = ~_near_edges(fw, kw)
    g = step.grad[idx].double().cpu().numpy()
    bad = (np.abs(g - g_ref) > GRAD_ATOL + GRAD_RTOL * np.abs(g_ref)) & keep[:, None, None]
    assert not bad.any(), (int(bad.sum()), tuple(np.argwhere(bad)[0]))


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_reference_argmax_ties(dtype):
    """The reference's greedy token is its first maximum.  Rows where x* holds the maximum
    together with an earlier element (same 16-byte vector, or an earlier one), only later
    elements, or alone: tau^ref must follow the lowest index exactly."""
    V = 4104
    target, draft, ref = _batch(2, 1, 8, 2, V, dtype, seed=9)
    x = target.float().argmax(-1)                       # x* per row (distinct values: no tie in z_p)
    rows = ref.view(-1, V)
    xs = x.view(-1)
    top = rows.float().amax(-1) + 4.0
    E = 16 // rows.element_size()
    for r in range(rows.shape[0]):
        k = int(xs[r])
        case = r % 4
        rows[r, k] = top[r]
        if case == 1 and k % E != 0:
            rows[r, k - 1] = top[r]                     # an earlier tie in the same vector
        elif case == 2 and k >= E:
            rows[r, k - E] = top[r]                     # an earlier tie in an earlier vector
        elif case == 3 and k + 1 < V:
            rows[r, k + 1] = top[r]                     # only a later tie: x* stays first
    N, K = draft.shape[:2]
    gp = dict(windows_per_rollout=1, rollouts_per_group=8)
    step = GrpoStep(target, draft, ref, aal.AAL_GRPO, dloss=float(N * K), **gp)
    rw = oracle.accept_reward(target.cpu(), draft.cpu(), ref.cpu(), 1, windows_per_rollout=1, rollouts_per_group=8)
    np.testing.assert_array_equal(step.tau_ref.cpu().numpy(), rw["tau_ref"])
    assert rw["tau_ref"].max() >= 1 and rw["tau_ref"].min() == 0
