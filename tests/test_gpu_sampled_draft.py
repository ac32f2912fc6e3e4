"""GPU parity of the sampled-draft reward (AAL_SAMPLING | AAL_SAMPLED_DRAFT): the drafted token is
drawn from q~ by Gumbel-max over counter-based uniforms, then accepted with probability
min(1, p~/q~) (Sec. 2.3).  tau is compared bit-exactly with the oracle, except on windows whose
leading run depends on a decision the kernel's fp32 arithmetic may take either way: a draw u
within 1e-5 of its threshold, or a Gumbel-max whose two best perturbed logits lie within 1e-4."""

import numpy as np
import pytest
import torch

import oracle
import paper_2609_24150_gb300 as aal
import synth
from tests.parity import note_thr
from tests.test_gpu_reward import run_reward

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
MODE = aal.AAL_SAMPLING | aal.AAL_SAMPLED_DRAFT
THR_BAND = 1e-5
KEY_BAND = 1e-4


def _gap(z, T, seed, n, k):
    """The margin of the Gumbel-max draw for window n, depth k (natural-log units)."""
    U = oracle.gumbel_uniforms(seed, n, k, z.shape[-1])
    key = z / T - np.log(-np.log(U))
    top = np.sort(key)[-2:]
    return top[1] - top[0]


def oracle_windows(target, draft, ref, T, seed, row_offset, windows):
    taus, taurs, amb = [], [], []
    for n in windows:
        t_h = target[n:n + 1].cpu()
        d_h = draft[n:n + 1].cpu()
        r_h = None if ref is None else ref[n:n + 1].cpu()
        o = oracle.accept_reward(t_h, d_h, r_h, oracle.REWARD_SAMPLED_DRAFT, T, seed, row_offset + int(n))
        taus.append(o["tau"][0])
        taurs.append(o["tau_ref"][0] if r_h is not None else 0)
        K = t_h.shape[1]
        a = False
        for thr, tau, z in ((o["thr"], o["tau"][0], d_h), (o["thr_ref"], taurs[-1], r_h)):
            if thr is None:
                continue
            upto = min(K, tau + 1)      # the depths whose decisions made the leading run
            a |= bool(np.any(np.abs(o["u"][0, :upto] - thr[0, :upto]) < THR_BAND))
            zz = oracle.as_f64(z)[0]
            a |= any(_gap(zz[k], T, seed, row_offset + int(n), k) < KEY_BAND for k in range(upto))
        amb.append(a)
    note_thr(int(np.sum(amb)), len(amb))
    return np.array(taus), np.array(taurs), np.array(amb)


@pytest.mark.parametrize("T", [1.0, 0.7])
@pytest.mark.parametrize("dtype,V", [(torch.float32, 1000), (torch.bfloat16, 4104), (torch.bfloat16, 7)])
@pytest.mark.parametrize("with_ref", [False, True])
def test_small_groups_all_windows(T, dtype, V, with_ref):
    wpr, rpg, groups, K = 2, 4, 2, 4
    target, draft, ref = synth.make_reward_logits(0, seed=3, with_ref=with_ref, windows_per_rollout=wpr,
                                                  rollouts_per_group=rpg * groups, K=K, V=V, dtype=dtype,
                                                  ref_from_draft=0.3)
    draft[::2] = target[::2]          # windows that accept often
    t, d = target.to(DEV), draft.to(DEV)
    r = None if ref is None else ref.to(DEV)
    got = run_reward(t, d, r, MODE, T, seed=11, row_offset=500, wpr=wpr, rpg=rpg, clip=3.0)
    N = t.shape[0]
    taus, taurs, amb = oracle_windows(t, d, r, T, 11, 500, range(N))
    keep = ~amb
    assert keep.sum() >= N - 2
    np.testing.assert_array_equal(got["tau"][keep], taus[keep])
    if r is not None:
        np.testing.assert_array_equal(got["tau_ref"][keep], taurs[keep])
    if keep.all():
        exp = oracle.accept_reward(target, draft, ref, oracle.REWARD_SAMPLED_DRAFT, T, 11, 500, wpr, rpg, 3.0)
        np.testing.assert_allclose(got["advantage"], exp["advantage"], rtol=0, atol=1e-5)
    assert got["tau"].max() >= 1


def test_full_prompt_group_mean_is_the_wtv_expected_length():
    """One reward group (4096 windows, K = 8, V = 128256 bf16): the mean of tau over the group
    equals the mean WTV expected length the loss forward reports for the same windows (5 standard
    errors), and sampled windows match the oracle exactly."""
    target, draft, _ = synth.make_reward_logits(0, seed=0, device=DEV)
    N, K, V = draft.shape
    T = 1.0
    got = run_reward(target, draft, None, MODE, T, seed=21, row_offset=0, wpr=256, rpg=16)
    prob = aal.loss_problem(draft, aal.AAL_SAMPLING, T, 0.0, 1.0)
    ws = torch.empty(aal.aal_workspace_size(prob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    eal = torch.empty(N, 2, device=DEV)
    aal.aal_loss_fwd(prob, draft, target, None, ws, loss, eal)
    es = eal[:, 1].double().cpu().numpy()
    tau = got["tau"].astype(np.float64)
    assert abs(tau.mean() - es.mean()) <= 5 * tau.std() / np.sqrt(N), (tau.mean(), es.mean())
    sel = [0, 1, 2049, N - 1]
    taus, _, amb = oracle_windows(target, draft, None, T, 21, 0, sel)
    keep = ~amb
    np.testing.assert_array_equal(got["tau"][sel][keep], taus[keep])


# ------------------------------------------------------------------ from a loss forward's normalisers

def run_sampled_from_loss(target, draft, T, seed, row_offset, wpr, rpg, clip=5.0, loss_mode=aal.AAL_BOTH):
    """aal_loss_fwd at T, then aal_accept_reward_sampled_from_loss over the same logits."""
    lprob = aal.loss_problem(draft, loss_mode, T, 0.5, 0.5)
    lws = torch.empty(aal.aal_workspace_size(lprob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    aal.aal_loss_fwd(lprob, draft, target, None, lws, loss)
    rprob = aal.reward_problem(draft, MODE, T, clip, seed, row_offset, wpr, rpg)
    rws = torch.empty(aal.aal_reward_workspace_size(rprob), dtype=torch.uint8, device=DEV)
    N = draft.shape[0]
    tau = torch.full((N,), -1, dtype=torch.int32, device=DEV)
    rl = torch.full((N // wpr,), float("nan"), device=DEV)
    adv = torch.full((N // wpr,), float("nan"), device=DEV)
    aal.aal_accept_reward_sampled_from_loss(rprob, lprob, draft, target, lws, rws, tau, rl, adv)
    torch.cuda.synchronize()
    assert aal.aal_check_device_status(rws) == aal.AAL_OK
    return dict(tau=tau.cpu().numpy(), rollout_len=rl.cpu().numpy(), advantage=adv.cpu().numpy())


@pytest.mark.parametrize("T", [1.0, 0.7])
@pytest.mark.parametrize("dtype,V", [(torch.float32, 1000), (torch.bfloat16, 4104), (torch.bfloat16, 7),
                                     (torch.bfloat16, 40000)])
def test_sampled_reward_from_loss_normalisers(T, dtype, V):
    """The draft streamed alone, the acceptance from the loss forward's normalisers: tau equals the
    oracle's and the logit pass's on every window whose decisions are not within rounding (V = 7
    rows are not 16-byte multiples and take the reward's own pass)."""
    wpr, rpg, groups, K = 2, 4, 2, 4
    target, draft, _ = synth.make_reward_logits(0, seed=5, windows_per_rollout=wpr, rollouts_per_group=rpg * groups,
                                                K=K, V=V, dtype=dtype)
    draft[::2] = target[::2]
    t, d = target.to(DEV), draft.to(DEV)
    got = run_sampled_from_loss(t, d, T, seed=13, row_offset=700, wpr=wpr, rpg=rpg, clip=3.0)
    logit = run_reward(t, d, None, MODE, T, seed=13, row_offset=700, wpr=wpr, rpg=rpg, clip=3.0)
    N = t.shape[0]
    taus, _, amb = oracle_windows(t, d, None, T, 13, 700, range(N))
    keep = ~amb
    assert keep.sum() >= N - 2
    np.testing.assert_array_equal(got["tau"][keep], taus[keep])
    np.testing.assert_array_equal(got["tau"][keep], logit["tau"][keep])
    if keep.all():
        np.testing.assert_allclose(got["advantage"], logit["advantage"], rtol=0, atol=1e-6)
    assert got["tau"].max() >= 1


def test_sampled_reward_from_loss_full_group():
    """One reward group (4096 windows, K = 8, V = 128256 bf16) after the WTV forward: tau equals the
    logit pass's on all but the windows a rounding can tip (at most 1%), and sampled windows
    match the oracle exactly."""
    target, draft, _ = synth.make_reward_logits(0, seed=0, device=DEV)
    N = draft.shape[0]
    T = 1.0
    got = run_sampled_from_loss(target, draft, T, seed=21, row_offset=0, wpr=256, rpg=16,
                                loss_mode=aal.AAL_SAMPLING)
    logit = run_reward(target, draft, None, MODE, T, seed=21, row_offset=0, wpr=256, rpg=16)
    differ = got["tau"] != logit["tau"]
    assert differ.mean() <= 0.01, differ.mean()
    sel = [0, 1, 2049, N - 1] + [int(i) for i in np.flatnonzero(differ)[:4]]
    taus, _, amb = oracle_windows(target, draft, None, T, 21, 0, sel)
    keep = ~amb
    np.testing.assert_array_equal(got["tau"][sel][keep], taus[keep])
    # a window where the two paths differ must be one the oracle calls ambiguous
    for j, n in enumerate(sel):
        if differ[n]:
            assert amb[j], n
