"""GPU parity of the GRPO acceptance reward against the oracle (through the C ABI).

tau is compared bit-exactly.  Under sampling verification a draw u that sits within
1e-5 of its threshold min(1, p~/q~) may be decided either way by the kernel's fp32
log-sum-exps (their error is a few 1e-6 in log2 units), so windows whose leading run
depends on such a draw are set aside (and with them their group's advantages).
"""

import numpy as np
import pytest
import torch

import oracle
import paper_2609_24150_gb300 as aal
import synth
from oracle.reward import REWARD_GREEDY, REWARD_SAMPLING
from tests.parity import assert_bands, note_thr

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
THR_BAND = 1e-5
OMODE = {aal.AAL_GREEDY: REWARD_GREEDY, aal.AAL_SAMPLING: REWARD_SAMPLING}


def run_reward(target, draft, ref, mode, T=1.0, seed=0, row_offset=0, wpr=1, rpg=1, clip=5.0):
    prob = aal.reward_problem(draft, mode, T, clip, seed, row_offset, wpr, rpg)
    ws = torch.empty(aal.aal_reward_workspace_size(prob), dtype=torch.uint8, device=DEV)
    N = draft.shape[0]
    tau = torch.full((N,), -1, dtype=torch.int32, device=DEV)
    tau_ref = torch.full((N,), -1, dtype=torch.int32, device=DEV)
    rl = torch.full((N // wpr,), float("nan"), device=DEV)
    adv = torch.full((N // wpr,), float("nan"), device=DEV)
    aal.aal_accept_reward(prob, draft, target, ref, ws, tau, tau_ref if ref is not None else None, rl, adv)
    torch.cuda.synchronize()
    assert aal.aal_check_device_status(ws) == aal.AAL_OK
    return dict(tau=tau.cpu().numpy(), tau_ref=tau_ref.cpu().numpy(), rollout_len=rl.cpu().numpy(),
                advantage=adv.cpu().numpy())


def oracle_chunked(target, draft, ref, mode, T, seed, row_offset, windows, chunk=16):
    """Oracle tau (and ambiguity flags) for the given windows, a few windows at a time."""
    taus, taurs, amb = [], [], []
    windows = np.asarray(windows)
    for c0 in range(0, len(windows), chunk):
        w = windows[c0:c0 + chunk]
        idx = torch.as_tensor(w, device=target.device)
        t_h = target[idx].cpu()
        d_h = draft[idx].cpu()
        r_h = None if ref is None else ref[idx].cpu()
        for j, n in enumerate(w):
            o = oracle.accept_reward(t_h[j:j + 1], d_h[j:j + 1], None if r_h is None else r_h[j:j + 1],
                                     OMODE[mode], T, seed, row_offset + int(n))
            taus.append(o["tau"][0])
            taurs.append(o["tau_ref"][0] if o["tau_ref"] is not None else 0)
            a = False
            if mode == aal.AAL_SAMPLING:
                K = t_h.shape[1]
                for thr, tau in ((o["thr"], o["tau"][0]), (o["thr_ref"], o["tau_ref"][0] if o["tau_ref"] is not None else None)):
                    if thr is None:
                        continue
                    upto = min(K, tau + 1)   # the draws that decided the leading run
                    a |= bool(np.any(np.abs(o["u"][0, :upto] - thr[0, :upto]) < THR_BAND))
            amb.append(a)
    note_thr(int(np.sum(amb)), len(amb))
    return np.array(taus), np.array(taurs), np.array(amb)


@pytest.mark.parametrize("mode,T", [(aal.AAL_GREEDY, 1.0), (aal.AAL_SAMPLING, 1.0), (aal.AAL_SAMPLING, 0.7)])
@pytest.mark.parametrize("dtype,V", [(torch.float32, 1000), (torch.bfloat16, 1001), (torch.bfloat16, 4096)])
@pytest.mark.parametrize("with_ref", [False, True])
def test_small_groups_all_windows(mode, T, dtype, V, with_ref):
    wpr, rpg, groups, K = 4, 4, 3, 8
    target, draft, ref = synth.make_reward_logits(0, seed=1, with_ref=with_ref, windows_per_rollout=wpr,
                                                  rollouts_per_group=rpg * groups, K=K, V=V, dtype=dtype)
    # make some windows agree with the target so the runs are not all zero
    draft[::3] = target[::3]
    t, d = target.to(DEV), draft.to(DEV)
    r = None if ref is None else ref.to(DEV)
    got = run_reward(t, d, r, mode, T, seed=5, row_offset=1000, wpr=wpr, rpg=rpg, clip=2.5)
    exp = oracle.accept_reward(target, draft, ref, OMODE[mode], T, 5, 1000, wpr, rpg, 2.5)
    N = t.shape[0]
    _, _, amb = oracle_chunked(t, d, r, mode, T, 5, 1000, np.arange(N))
    keep = ~amb
    np.testing.assert_array_equal(got["tau"][keep], exp["tau"][keep])
    if ref is not None:
        np.testing.assert_array_equal(got["tau_ref"][keep], exp["tau_ref"][keep])
    if keep.all():
        np.testing.assert_allclose(got["rollout_len"], exp["rollout_len"], rtol=0, atol=1e-6)
        np.testing.assert_allclose(got["advantage"], exp["advantage"], rtol=0, atol=1e-5)
        assert np.all(np.abs(got["advantage"]) <= 2.5)


def test_identical_drafts_accept_everything_greedy():
    target, _, _ = synth.make_reward_logits(0, windows_per_rollout=2, rollouts_per_group=2, K=5, V=300)
    t = target.to(DEV)
    got = run_reward(t, t.clone(), t.clone(), aal.AAL_GREEDY, wpr=2, rpg=2)
    assert np.all(got["tau"] == 5) and np.all(got["tau_ref"] == 5)
    assert np.all(got["rollout_len"] == 0) and np.all(got["advantage"] == 0)


def test_philox_draws_match_oracle_bit_exactly():
    """With p = q every sampled draft token has threshold 1, so tau = K whatever u is; with a
    draft that puts q~(S) = 2 p~(S) the threshold is 1/2 and accept == (u < 1/2) exposes u's bit."""
    K, V, N = 8, 64, 512
    target = torch.zeros(N, K, V)
    target[..., 0] = 1.0                      # p~(0) = e/(e + 63)
    draft = target.clone()
    # choose the draft logit at 0 so that q~(0) = 2 p~(0) exactly in fp64 terms
    p0 = np.e / (np.e + V - 1)
    q0 = 2 * p0
    draft[..., 0] = float(np.log(q0 * (V - 1) / (1 - q0)))
    t, d = target.to(DEV), draft.to(DEV)
    got = run_reward(t, d, None, aal.AAL_SAMPLING, 1.0, seed=123456789, row_offset=77)
    exp = oracle.accept_reward(target, draft, None, REWARD_SAMPLING, 1.0, 123456789, 77)
    keep = np.ones(N, dtype=bool)
    for n in range(N):
        upto = min(K, exp["tau"][n] + 1)
        keep[n] = not np.any(np.abs(exp["u"][n, :upto] - exp["thr"][n, :upto]) < THR_BAND)
    np.testing.assert_array_equal(got["tau"][keep], exp["tau"][keep])
    assert keep.mean() > 0.99


@pytest.fixture(scope="module")
def reward_group():
    target, draft, ref = synth.make_reward_logits(1, seed=0, device=DEV, with_ref=True)
    yield target, draft, ref
    del target, draft, ref
    torch.cuda.empty_cache()


@pytest.mark.parametrize("mode", [aal.AAL_GREEDY, aal.AAL_SAMPLING])
def test_full_prompt_group_sampled_windows(reward_group, mode):
    """One full prompt group (16 rollouts x 256 windows, K=8, V=128256 bf16) as streamed by the
    benchmark, with the global row offset of group 1; windows sampled for the oracle (400 under
    sampling verification, so that the share the threshold band sets aside is bounded)."""
    target, draft, ref = reward_group
    N = target.shape[0]
    got = run_reward(target, draft, ref, mode, 1.0, seed=0, row_offset=N, wpr=256, rpg=16)
    rng = np.random.default_rng(2)
    nsample = 46 if mode == aal.AAL_GREEDY else 400
    windows = np.array(sorted(set([0, N - 1] + list(rng.choice(N, nsample, replace=False)))))
    tau, taur, amb = oracle_chunked(target, draft, ref, mode, 1.0, 0, N, windows)
    assert_bands()
    keep = ~amb
    np.testing.assert_array_equal(got["tau"][windows][keep], tau[keep])
    np.testing.assert_array_equal(got["tau_ref"][windows][keep], taur[keep])
    # advantages are standardised within the group and clipped
    A = got["advantage"]
    assert abs(A.mean()) < 1e-5 and np.all(np.abs(A) <= 5.0)
    rl = got["rollout_len"]
    R = got["tau"].astype(np.float64) - got["tau_ref"]
    np.testing.assert_allclose(rl, R.reshape(16, 256).mean(1), atol=1e-6)


@pytest.mark.parametrize("dtype,V", [(torch.float32, 1000), (torch.bfloat16, 1001), (torch.bfloat16, 4096),
                                     (torch.bfloat16, 32000), (torch.bfloat16, 8200)])
@pytest.mark.parametrize("mode,T", [(aal.AAL_GREEDY, 1.0), (aal.AAL_SAMPLING, 1.0), (aal.AAL_SAMPLING, 0.7)])
def test_reward_from_loss_statistics(dtype, V, mode, T):
    """The reward taken from a loss forward's statistics equals the one from a logit pass
    (greedy bit-exactly; sampling apart from draws on the threshold) and the oracle's."""
    wpr, rpg = 4, 4
    target, draft, _ = synth.make_reward_logits(0, seed=V, windows_per_rollout=wpr, rollouts_per_group=rpg * 2,
                                                K=6, V=V, dtype=dtype)
    draft[::3] = target[::3]
    t, d = target.to(DEV), draft.to(DEV)
    N = t.shape[0]
    lprob = aal.loss_problem(d, aal.AAL_BOTH, T, 0.5, 0.5)
    lws = torch.empty(aal.aal_workspace_size(lprob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    aal.aal_loss_fwd(lprob, d, t, None, lws, loss)
    rprob = aal.reward_problem(d, mode, T, 2.0, 17, 5000, wpr, rpg)
    rws = torch.empty(aal.aal_reward_workspace_size(rprob), dtype=torch.uint8, device=DEV)
    tau = torch.full((N,), -1, dtype=torch.int32, device=DEV)
    rl = torch.full((N // wpr,), float("nan"), device=DEV)
    adv = torch.full((N // wpr,), float("nan"), device=DEV)
    aal.aal_accept_reward_from_loss(rprob, lprob, lws, rws, tau, rl, adv)
    torch.cuda.synchronize()
    got = dict(tau=tau.cpu().numpy(), rollout_len=rl.cpu().numpy(), advantage=adv.cpu().numpy())
    logit = run_reward(t, d, None, mode, T, seed=17, row_offset=5000, wpr=wpr, rpg=rpg, clip=2.0)
    exp = oracle.accept_reward(target, draft, None, OMODE[mode], T, 17, 5000, wpr, rpg, 2.0)
    _, _, amb = oracle_chunked(t, d, None, mode, T, 17, 5000, np.arange(N))
    keep = ~amb
    np.testing.assert_array_equal(got["tau"][keep], exp["tau"][keep])
    np.testing.assert_array_equal(got["tau"][keep], logit["tau"][keep])
    if keep.all():
        np.testing.assert_allclose(got["rollout_len"], exp["rollout_len"], rtol=0, atol=1e-6)
        np.testing.assert_allclose(got["advantage"], exp["advantage"], rtol=0, atol=1e-5)


def test_reward_from_loss_full_size_greedy():
    """The bench's configuration: V=128256 bf16, 8192 windows of K=7, after the EAL+WTV forward."""
    target, draft, _ = synth.make_logits("v128k", seed=3, device=DEV)
    N = target.shape[0]
    lprob = aal.loss_problem(draft, aal.AAL_BOTH, 1.0, 0.5, 0.5)
    lws = torch.empty(aal.aal_workspace_size(lprob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    aal.aal_loss_fwd(lprob, draft, target, None, lws, loss)
    rprob = aal.reward_problem(draft, aal.AAL_GREEDY, 1.0, 5.0, 0, 0, 256, 16)
    rws = torch.empty(aal.aal_reward_workspace_size(rprob), dtype=torch.uint8, device=DEV)
    tau = torch.empty(N, dtype=torch.int32, device=DEV)
    rl = torch.empty(N // 256, device=DEV)
    adv = torch.empty(N // 256, device=DEV)
    aal.aal_accept_reward_from_loss(rprob, lprob, lws, rws, tau, rl, adv)
    logit = run_reward(target, draft, None, aal.AAL_GREEDY, wpr=256, rpg=16)
    np.testing.assert_array_equal(tau.cpu().numpy(), logit["tau"])
    np.testing.assert_array_equal(adv.cpu().numpy(), logit["advantage"])
    # sampled windows against the oracle
    rng = np.random.default_rng(4)
    windows = np.array(sorted(set([0, N - 1] + list(rng.choice(N, 30, replace=False)))))
    tau_o, _, _ = oracle_chunked(target, draft, None, aal.AAL_GREEDY, 1.0, 0, 0, windows)
    np.testing.assert_array_equal(tau.cpu().numpy()[windows], tau_o)
    del target, draft
    torch.cuda.empty_cache()
