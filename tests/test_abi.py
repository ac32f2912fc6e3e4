"""The C-ABI library loads, exports what include/aal.h declares, and rejects bad arguments
on the host before launching anything (CPU only: no call here reaches the GPU)."""

import ctypes
import glob
import os
import re
import subprocess

import pytest
import torch

import paper_2609_24150_gb300 as aal

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        names |= set(re.findall(r"AAL_API\s+[\w\s\*]+?\b(aal_\w+)\s*\(", text))
    return names


def test_header_declares_the_entry_points():
    names = _declared()
    assert {"aal_loss_fwd", "aal_loss_bwd", "aal_loss_fwd_bwd", "aal_seq_loss_fwd", "aal_seq_loss_bwd",
            "aal_seq_loss_fwd_bwd", "aal_accept_reward", "aal_workspace_size",
            "aal_reward_workspace_size", "aal_check_device_status", "aal_status_string",
            "aal_abi_version"} <= names


def test_library_exports_every_declared_symbol():
    lib = aal.library()
    for name in _declared():
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", aal.library_path()], capture_output=True,
                         text=True).stdout
    exported = {l.split()[-1] for l in out.splitlines() if " T " in l}
    assert {n for n in exported if n.startswith("aal_")} == _declared()


def test_status_strings_and_version():
    assert aal.aal_abi_version() == 10700
    for code in range(6):
        assert aal.aal_status_string(code).startswith("AAL_")
    assert aal.aal_status_string(99) == "unknown aal_status"


def _prob(**kw):
    d = dict(N=4, K=3, V=100, dtype=aal.AAL_BF16, mode=aal.AAL_BOTH, temperature=1.0,
             w_greedy=0.5, w_sampling=0.5, w_kl=1.0, w_tv=0.1, global_counts=0)
    d.update(kw)
    return aal.AalProblem(**d)


def _ws_size(p):
    out = ctypes.c_size_t(0)
    code = aal.library().aal_workspace_size(ctypes.byref(p), ctypes.byref(out))
    return code, out.value


def test_workspace_size_grows_with_rows():
    c1, s1 = _ws_size(_prob(N=4))
    c2, s2 = _ws_size(_prob(N=4096))
    assert c1 == c2 == aal.AAL_OK and 0 < s1 < s2 and s1 % 256 == 0


@pytest.mark.parametrize("kw,code", [
    (dict(K=0), aal.AAL_ERR_INVALID_ARG),
    (dict(K=9), aal.AAL_ERR_UNSUPPORTED),
    (dict(V=0), aal.AAL_ERR_INVALID_ARG),
    (dict(N=-1), aal.AAL_ERR_INVALID_ARG),
    (dict(dtype=7), aal.AAL_ERR_INVALID_ARG),
    (dict(mode=0), aal.AAL_ERR_INVALID_ARG),
    (dict(mode=64), aal.AAL_ERR_INVALID_ARG),
    (dict(mode=aal.AAL_IDS | aal.AAL_GREEDY), aal.AAL_OK),
    (dict(mode=aal.AAL_IDS | aal.AAL_GRPO), aal.AAL_OK),
    (dict(mode=aal.AAL_IDS), aal.AAL_ERR_INVALID_ARG),
    (dict(mode=aal.AAL_IDS | aal.AAL_BOTH), aal.AAL_ERR_INVALID_ARG),
    (dict(mode=aal.AAL_IDS | aal.AAL_GREEDY | aal.AAL_KL), aal.AAL_ERR_INVALID_ARG),
    (dict(mode=aal.AAL_IDS | aal.AAL_GREEDY | aal.AAL_TV), aal.AAL_ERR_INVALID_ARG),
    (dict(mode=aal.AAL_KL | aal.AAL_TV), aal.AAL_OK),
    (dict(mode=aal.AAL_TV, temperature=0.0), aal.AAL_ERR_INVALID_ARG),
    (dict(w_tv=float("inf")), aal.AAL_ERR_INVALID_ARG),
    (dict(mode=aal.AAL_GRPO | aal.AAL_KL | aal.AAL_GREEDY), aal.AAL_OK),
    (dict(mode=-1), aal.AAL_ERR_INVALID_ARG),
    (dict(w_kl=float("nan")), aal.AAL_ERR_INVALID_ARG),
    (dict(temperature=0.0), aal.AAL_ERR_INVALID_ARG),
    (dict(temperature=-1.0), aal.AAL_ERR_INVALID_ARG),
    (dict(temperature=float("nan")), aal.AAL_ERR_INVALID_ARG),
    (dict(w_greedy=float("inf")), aal.AAL_ERR_INVALID_ARG),
    (dict(global_counts=2), aal.AAL_ERR_INVALID_ARG),
    (dict(global_counts=-1), aal.AAL_ERR_INVALID_ARG),
    (dict(global_counts=1, n_windows_global=10, n_positions_global=30), aal.AAL_OK),
    (dict(global_counts=1, n_windows_global=0, n_positions_global=0), aal.AAL_OK),
    (dict(global_counts=1, n_windows_global=-1, n_positions_global=30), aal.AAL_ERR_INVALID_ARG),
    (dict(global_counts=1, n_windows_global=10, n_positions_global=2**31), aal.AAL_ERR_INVALID_ARG),
    (dict(global_counts=0, n_windows_global=-5, n_positions_global=-5), aal.AAL_OK),  # not read
    (dict(V=2**31), aal.AAL_ERR_UNSUPPORTED),
    (dict(N=2**60, V=2**20), aal.AAL_ERR_INVALID_ARG),
])
def test_bad_problems_are_rejected(kw, code):
    assert _ws_size(_prob(**kw))[0] == code


def test_greedy_mode_accepts_zero_temperature():
    assert _ws_size(_prob(mode=aal.AAL_GREEDY, temperature=0.0))[0] == aal.AAL_OK
    assert _ws_size(_prob(mode=aal.AAL_GREEDY | aal.AAL_KL, temperature=0.0))[0] == aal.AAL_OK
    assert _ws_size(_prob(mode=aal.AAL_KL, temperature=0.0))[0] == aal.AAL_OK
    assert _ws_size(_prob(mode=aal.AAL_KL | aal.AAL_SAMPLING, temperature=0.0))[0] == aal.AAL_ERR_INVALID_ARG


def test_null_and_misaligned_pointers_rejected_before_launch():
    lib = aal.library()
    p = _prob()
    code, size = _ws_size(p)
    fake_ws = 1 << 20                      # never dereferenced: rejected before any launch
    fake = 1 << 24
    # NULL problem
    assert lib.aal_loss_fwd(None, fake, fake, None, fake_ws, size, fake, None, None) == aal.AAL_ERR_INVALID_ARG
    # NULL / misaligned logits
    assert lib.aal_loss_fwd(ctypes.byref(p), None, fake, None, fake_ws, size, fake, None, None) == aal.AAL_ERR_INVALID_ARG
    assert lib.aal_loss_fwd(ctypes.byref(p), fake + 2, fake, None, fake_ws, size, fake, None, None) == aal.AAL_ERR_INVALID_ARG
    # NULL loss
    assert lib.aal_loss_fwd(ctypes.byref(p), fake, fake, None, fake_ws, size, None, None, None) == aal.AAL_ERR_INVALID_ARG
    # workspace too small / misaligned / missing
    assert lib.aal_loss_fwd(ctypes.byref(p), fake, fake, None, fake_ws, size - 1, fake, None, None) == aal.AAL_ERR_WORKSPACE
    assert lib.aal_loss_fwd(ctypes.byref(p), fake, fake, None, fake_ws + 16, size, fake, None, None) == aal.AAL_ERR_WORKSPACE
    assert lib.aal_loss_fwd(ctypes.byref(p), fake, fake, None, None, size, fake, None, None) == aal.AAL_ERR_WORKSPACE
    # backward: NULL gradient, non-finite upstream gradient
    assert lib.aal_loss_bwd(ctypes.byref(p), fake, fake, None, fake_ws, size, 1.0, None, None) == aal.AAL_ERR_INVALID_ARG
    assert lib.aal_loss_bwd(ctypes.byref(p), fake, fake, None, fake_ws, size, float("nan"), fake, None) == aal.AAL_ERR_INVALID_ARG
    # the one-call forward + backward: every check of both calls, and GRPO refused
    fb = lambda prob, d=fake, ws=fake_ws, sz=size, dl=1.0, loss=fake, grad=fake: lib.aal_loss_fwd_bwd(
        ctypes.byref(prob), d, fake, None, ws, sz, dl, loss, None, grad, None)
    assert fb(p, grad=None) == aal.AAL_ERR_INVALID_ARG
    assert fb(p, loss=None) == aal.AAL_ERR_INVALID_ARG
    assert fb(p, d=fake + 2) == aal.AAL_ERR_INVALID_ARG
    assert fb(p, dl=float("inf")) == aal.AAL_ERR_INVALID_ARG
    assert fb(p, sz=size - 1) == aal.AAL_ERR_WORKSPACE
    assert fb(_prob(mode=aal.AAL_GRPO | aal.AAL_GREEDY)) == aal.AAL_ERR_UNSUPPORTED
    assert fb(_prob(K=9)) == aal.AAL_ERR_UNSUPPORTED


def _rprob(**kw):
    d = dict(N=8, K=4, V=100, dtype=aal.AAL_BF16, mode=aal.AAL_GREEDY, temperature=1.0,
             adv_clip=5.0, seed=0, row_offset=0, windows_per_rollout=2, rollouts_per_group=2)
    d.update(kw)
    return aal.AalRewardProblem(**d)


@pytest.mark.parametrize("kw,code", [
    (dict(), aal.AAL_OK),
    (dict(mode=aal.AAL_BOTH), aal.AAL_ERR_INVALID_ARG),
    (dict(mode=aal.AAL_SAMPLING, temperature=0.0), aal.AAL_ERR_INVALID_ARG),
    (dict(mode=aal.AAL_SAMPLING | aal.AAL_SAMPLED_DRAFT), aal.AAL_OK),
    (dict(mode=aal.AAL_GREEDY | aal.AAL_SAMPLED_DRAFT), aal.AAL_ERR_INVALID_ARG),
    (dict(mode=aal.AAL_SAMPLED_DRAFT), aal.AAL_ERR_INVALID_ARG),
    (dict(windows_per_rollout=3), aal.AAL_ERR_INVALID_ARG),     # 8 windows not a multiple of 6
    (dict(rollouts_per_group=0), aal.AAL_ERR_INVALID_ARG),
    (dict(adv_clip=0.0), aal.AAL_ERR_INVALID_ARG),
    (dict(row_offset=-1), aal.AAL_ERR_INVALID_ARG),
    (dict(K=9), aal.AAL_ERR_UNSUPPORTED),
])
def test_reward_problem_checks(kw, code):
    out = ctypes.c_size_t(0)
    p = _rprob(**kw)
    assert aal.library().aal_reward_workspace_size(ctypes.byref(p), ctypes.byref(out)) == code


def test_binding_refuses_cpu_tensors():
    t = torch.zeros(2, 2, 8, dtype=torch.bfloat16)
    p = aal.loss_problem(t, aal.AAL_BOTH)
    with pytest.raises(ValueError, match="CUDA"):
        aal.aal_loss_fwd(p, t, t, None, torch.zeros(1024, dtype=torch.uint8),
                         torch.zeros(1), None)


def test_reward_from_loss_argument_checks():
    lib = aal.library()
    lp = _prob(N=8, K=4, V=100, mode=aal.AAL_GREEDY, temperature=0.0)
    code, lsize = _ws_size(lp)
    rp = _rprob(N=8, K=4, V=100)
    fake = 1 << 24
    out = ctypes.c_size_t(0)
    assert lib.aal_reward_workspace_size(ctypes.byref(rp), ctypes.byref(out)) == 0
    rsize = out.value
    call = lambda r, l, lws=fake, lb=lsize: lib.aal_accept_reward_from_loss(
        ctypes.byref(r), ctypes.byref(l), lws, lb, fake, rsize, fake, fake, fake, None)
    # shapes must match the loss problem
    assert call(_rprob(N=8, K=4, V=101), lp) == aal.AAL_ERR_INVALID_ARG
    # sampling acceptance needs a loss with the sampling term at the same temperature
    assert call(_rprob(N=8, K=4, V=100, mode=aal.AAL_SAMPLING), lp) == aal.AAL_ERR_INVALID_ARG
    lps = _prob(N=8, K=4, V=100, mode=aal.AAL_BOTH, temperature=0.9)
    assert call(_rprob(N=8, K=4, V=100, mode=aal.AAL_SAMPLING, temperature=1.0), lps) == aal.AAL_ERR_INVALID_ARG
    # the loss workspace must be large enough
    assert call(rp, lp, fake, lsize - 1) == aal.AAL_ERR_WORKSPACE
    # a sampled draft needs the logits: the other entry point
    assert call(_rprob(N=8, K=4, V=100, mode=aal.AAL_SAMPLING | aal.AAL_SAMPLED_DRAFT), lps) == aal.AAL_ERR_INVALID_ARG


def test_sampled_reward_from_loss_argument_checks():
    lib = aal.library()
    SD = aal.AAL_SAMPLING | aal.AAL_SAMPLED_DRAFT
    lp = _prob(N=8, K=4, V=104, mode=aal.AAL_BOTH, temperature=0.8)
    code, lsize = _ws_size(lp)
    rp = _rprob(N=8, K=4, V=104, mode=SD, temperature=0.8)
    fake = 1 << 24
    out = ctypes.c_size_t(0)
    assert lib.aal_reward_workspace_size(ctypes.byref(rp), ctypes.byref(out)) == 0
    rsize = out.value
    call = lambda r, l, d=fake, t=fake, lb=lsize, rb=rsize: lib.aal_accept_reward_sampled_from_loss(
        ctypes.byref(r), ctypes.byref(l), d, t, fake, lb, fake, rb, fake, fake, fake, None)
    assert call(_rprob(N=8, K=4, V=104, mode=aal.AAL_SAMPLING, temperature=0.8), lp) == aal.AAL_ERR_INVALID_ARG
    assert call(_rprob(N=8, K=4, V=100, mode=SD, temperature=0.8), lp) == aal.AAL_ERR_INVALID_ARG
    assert call(rp, _prob(N=8, K=4, V=104, mode=aal.AAL_GREEDY, temperature=0.8)) == aal.AAL_ERR_INVALID_ARG
    assert call(rp, _prob(N=8, K=4, V=104, mode=aal.AAL_BOTH, temperature=1.0)) == aal.AAL_ERR_INVALID_ARG
    assert call(rp, lp, d=None) == aal.AAL_ERR_INVALID_ARG
    assert call(rp, lp, t=fake + 8) == aal.AAL_ERR_INVALID_ARG
    assert call(rp, lp, lb=lsize - 1) == aal.AAL_ERR_WORKSPACE
    assert call(rp, lp, rb=rsize - 1) == aal.AAL_ERR_WORKSPACE


def _sprob(**kw):
    d = dict(B=2, seq_len=16, K=4, V=100, dtype=aal.AAL_BF16, mode=aal.AAL_BOTH, temperature=1.0,
             w_greedy=0.5, w_sampling=0.5, w_kl=1.0, w_tv=0.1, full_windows=0, global_counts=0)
    d.update(kw)
    return aal.AalSeqProblem(**d)


def _seq_ws(p):
    out = ctypes.c_size_t(0)
    return aal.library().aal_seq_workspace_size(ctypes.byref(p), ctypes.byref(out)), out.value


@pytest.mark.parametrize("kw,code", [
    (dict(), aal.AAL_OK),
    (dict(B=0), aal.AAL_OK),
    (dict(seq_len=0), aal.AAL_OK),
    (dict(K=20), aal.AAL_ERR_UNSUPPORTED),
    (dict(K=0), aal.AAL_ERR_INVALID_ARG),
    (dict(B=-1), aal.AAL_ERR_INVALID_ARG),
    (dict(seq_len=-3), aal.AAL_ERR_INVALID_ARG),
    (dict(B=2**40, seq_len=2**40), aal.AAL_ERR_INVALID_ARG),     # B * seq_len overflows
    (dict(B=2**30, seq_len=2**20, V=2**20), aal.AAL_ERR_INVALID_ARG),  # logit bytes overflow
    (dict(V=0), aal.AAL_ERR_INVALID_ARG),
    (dict(mode=0), aal.AAL_ERR_INVALID_ARG),
    (dict(temperature=0.0), aal.AAL_ERR_INVALID_ARG),
    (dict(global_counts=2), aal.AAL_ERR_INVALID_ARG),
    (dict(global_counts=1, n_windows_global=64, n_positions_global=64), aal.AAL_OK),
    (dict(global_counts=1, n_windows_global=2**31, n_positions_global=64), aal.AAL_ERR_INVALID_ARG),
    (dict(full_windows=1), aal.AAL_OK),
    (dict(full_windows=2), aal.AAL_ERR_INVALID_ARG),
])
def test_seq_problem_checks(kw, code):
    assert _seq_ws(_sprob(**kw))[0] == code


def test_seq_workspace_holds_per_depth_partials():
    c1, s1 = _seq_ws(_sprob(K=1))
    c8, s8 = _seq_ws(_sprob(K=8))
    # two float[B*seq_len][K] arrays, each 256-byte aligned: 2 x (32*8*4 - 256) more bytes for K = 8
    assert c1 == c8 == aal.AAL_OK and s8 - s1 == 2 * (32 * 8 * 4 - 256) and s1 % 256 == 0


def test_seq_pointer_checks_before_launch():
    lib = aal.library()
    p = _sprob()
    code, size = _seq_ws(p)
    fake_ws, fake = 1 << 20, 1 << 24
    assert lib.aal_seq_loss_fwd(ctypes.byref(p), None, fake, None, fake_ws, size, fake, None, None) == aal.AAL_ERR_INVALID_ARG
    assert lib.aal_seq_loss_fwd(ctypes.byref(p), fake, fake + 8, None, fake_ws, size, fake, None, None) == aal.AAL_ERR_INVALID_ARG
    assert lib.aal_seq_loss_fwd(ctypes.byref(p), fake, fake, None, fake_ws, size, None, None, None) == aal.AAL_ERR_INVALID_ARG
    assert lib.aal_seq_loss_fwd(ctypes.byref(p), fake, fake, None, fake_ws, size - 1, fake, None, None) == aal.AAL_ERR_WORKSPACE
    assert lib.aal_seq_loss_bwd(ctypes.byref(p), fake, fake, None, fake_ws, size, 1.0, None, None) == aal.AAL_ERR_INVALID_ARG
    assert lib.aal_seq_loss_bwd(ctypes.byref(p), fake, fake, None, fake_ws, size, float("inf"), fake, None) == aal.AAL_ERR_INVALID_ARG
    assert lib.aal_seq_loss_bwd(ctypes.byref(p), fake, fake, None, fake_ws + 128, size, 1.0, fake, None) == aal.AAL_ERR_WORKSPACE
    fb = lib.aal_seq_loss_fwd_bwd
    assert fb(ctypes.byref(p), fake, fake, None, fake_ws, size, 1.0, fake, None, None, None) == aal.AAL_ERR_INVALID_ARG
    assert fb(ctypes.byref(p), fake, fake, None, fake_ws, size, 1.0, None, None, fake, None) == aal.AAL_ERR_INVALID_ARG
    assert fb(ctypes.byref(p), fake, fake + 8, None, fake_ws, size, 1.0, fake, None, fake, None) == aal.AAL_ERR_INVALID_ARG
    assert fb(ctypes.byref(p), fake, fake, None, fake_ws, size, float("nan"), fake, None, fake, None) == aal.AAL_ERR_INVALID_ARG
    assert fb(ctypes.byref(p), fake, fake, None, fake_ws, size - 1, 1.0, fake, None, fake, None) == aal.AAL_ERR_WORKSPACE
    g = _sprob(mode=aal.AAL_GREEDY | aal.AAL_GRPO)
    assert fb(ctypes.byref(g), fake, fake, None, fake_ws, _seq_ws(g)[1], 1.0, fake, None, fake, None) == aal.AAL_ERR_UNSUPPORTED


def _gprob(**kw):
    d = dict(N=8, K=4, V=100, dtype=aal.AAL_BF16, reserved=0, windows_per_rollout=1, rollouts_per_group=4,
             adv_clip=5.0, eps_clip=0.2, rho_min=0.0, rho_max=10.0, log_rho_clip=10.0, w_grpo=0.1)
    d.update(kw)
    return aal.AalGrpoProblem(**d)


@pytest.mark.parametrize("kw,code", [
    (dict(), aal.AAL_OK),
    (dict(rollouts_per_group=3), aal.AAL_ERR_INVALID_ARG),      # 8 windows not a multiple of 3
    (dict(eps_clip=1.0), aal.AAL_ERR_INVALID_ARG),
    (dict(eps_clip=-0.1), aal.AAL_ERR_INVALID_ARG),
    (dict(rho_min=2.0, rho_max=1.0), aal.AAL_ERR_INVALID_ARG),
    (dict(rho_min=-1.0), aal.AAL_ERR_INVALID_ARG),
    (dict(rho_max=float("inf")), aal.AAL_ERR_INVALID_ARG),
    (dict(log_rho_clip=0.0), aal.AAL_ERR_INVALID_ARG),
    (dict(w_grpo=float("nan")), aal.AAL_ERR_INVALID_ARG),
    (dict(adv_clip=0.0), aal.AAL_ERR_INVALID_ARG),
    (dict(reserved=1), aal.AAL_ERR_INVALID_ARG),
    (dict(K=9), aal.AAL_ERR_UNSUPPORTED),
])
def test_grpo_problem_checks(kw, code):
    out = ctypes.c_size_t(0)
    p = _gprob(**kw)
    assert aal.library().aal_grpo_workspace_size(ctypes.byref(p), ctypes.byref(out)) == code


def test_grpo_needs_a_matching_loss_problem_with_the_grpo_bit():
    lib = aal.library()
    g = _gprob()
    fake, fake_ws = 1 << 24, 1 << 20
    big = 1 << 30
    lp = _prob(N=8, K=4, mode=aal.AAL_GREEDY)                       # no AAL_GRPO bit
    assert lib.aal_grpo_from_loss(ctypes.byref(g), ctypes.byref(lp), fake_ws, big, fake, fake_ws, big,
                                  fake, None, None, None, None, None) == aal.AAL_ERR_INVALID_ARG
    lp = _prob(N=8, K=3, mode=aal.AAL_GREEDY | aal.AAL_GRPO)        # shape differs
    assert lib.aal_grpo_from_loss(ctypes.byref(g), ctypes.byref(lp), fake_ws, big, fake, fake_ws, big,
                                  fake, None, None, None, None, None) == aal.AAL_ERR_INVALID_ARG
    lp = _prob(N=8, K=4, mode=aal.AAL_GREEDY | aal.AAL_GRPO)
    assert lib.aal_grpo_from_loss(ctypes.byref(g), ctypes.byref(lp), fake_ws, big, None, fake_ws, big,
                                  fake, None, None, None, None, None) == aal.AAL_ERR_INVALID_ARG
    assert lib.aal_grpo_from_loss(ctypes.byref(g), ctypes.byref(lp), fake_ws, big, fake, fake_ws, big,
                                  None, None, None, None, None, None) == aal.AAL_ERR_INVALID_ARG
    assert lib.aal_grpo_from_loss(ctypes.byref(g), ctypes.byref(lp), fake_ws, 16, fake, fake_ws, big,
                                  fake, None, None, None, None, None) == aal.AAL_ERR_WORKSPACE
    assert lib.aal_grpo_from_loss(ctypes.byref(g), ctypes.byref(lp), fake_ws, big, fake, fake_ws, 16,
                                  fake, None, None, None, None, None) == aal.AAL_ERR_WORKSPACE


def test_sequence_grpo_checks():
    lib = aal.library()
    sp = _sprob(B=2, seq_len=16, K=4, mode=aal.AAL_GREEDY | aal.AAL_GRPO)
    assert _seq_ws(sp)[0] == aal.AAL_OK
    g = _gprob(N=8, K=4)
    out = ctypes.c_size_t(0)
    assert lib.aal_seq_grpo_workspace_size(ctypes.byref(g), ctypes.byref(sp), ctypes.byref(out)) == aal.AAL_OK
    size = out.value
    fake, fake_ws, big = 1 << 24, 1 << 20, 1 << 30
    args = lambda gp, spp, starts, ws_bytes: (ctypes.byref(gp), ctypes.byref(spp), fake_ws, big, fake, starts,
                                              fake_ws, ws_bytes, fake, None, None, None, None, None)
    assert lib.aal_seq_grpo_from_loss(*args(g, sp, None, size)) == aal.AAL_ERR_INVALID_ARG      # no starts
    assert lib.aal_seq_grpo_from_loss(*args(g, sp, fake + 2, size)) == aal.AAL_ERR_INVALID_ARG  # misaligned
    assert lib.aal_seq_grpo_from_loss(*args(g, sp, fake, size - 1)) == aal.AAL_ERR_WORKSPACE
    assert lib.aal_seq_grpo_from_loss(*args(_gprob(N=8, K=3), sp, fake, size)) == aal.AAL_ERR_INVALID_ARG
    no_grpo = _sprob(B=2, seq_len=16, K=4, mode=aal.AAL_GREEDY)
    assert lib.aal_seq_grpo_from_loss(*args(g, no_grpo, fake, size)) == aal.AAL_ERR_INVALID_ARG


def _launch_rows(N, K, G, S, m):
    """Row times of the fused launch: G groups take the first N - m S windows, one per row time
    each; S solo CTAs take m windows each, K row times per window."""
    return max(-(-(N - m * S) // G), m * K)


@pytest.mark.parametrize("K", [1, 2, 3, 4, 5, 6, 7, 8])
def test_solo_window_split_is_optimal(K):
    """The fused call's split of windows between CTA groups and solo CTAs, against a brute
    force over every m, for the SM count of a GB300 and of smaller parts."""
    for ctas in (152, 148, 132, 64, 13):
        for N in list(range(0, 400)) + [1000, 4096, 8191, 8192, 8193, 65536, 10**6 + 7]:
            G = min(ctas // K, N, 1024)
            S = ctas - G * K
            m = aal.aal_debug_solo_windows(N, K, G, S)
            if G <= 0 or S <= 0:
                assert m == 0
                continue
            assert 0 <= m and m * S <= N
            lo, hi = max(0, N // (G * K + S) - 3), min(N // S, N // (G * K + S) + 3)
            best = min(_launch_rows(N, K, G, S, j) for j in [0] + list(range(lo, hi + 1)))
            if N <= 400:   # the whole range as well, not just around the balance point
                best = min(best, min(_launch_rows(N, K, G, S, j) for j in range(0, N // S + 1)))
            assert _launch_rows(N, K, G, S, m) == best, (N, K, ctas, m)
            if _launch_rows(N, K, G, S, 0) == best:
                assert m == 0, (N, K, ctas, m)



def test_problem_struct_layout():
    """The ctypes mirrors have the header's layout: the data-parallel fields follow the int32 that
    was "reserved" before ABI 1.6 (so a caller that zeroes it never has them read)."""
    P, S = aal.AalProblem, aal.AalSeqProblem
    assert P.global_counts.offset == 52 and P.n_windows_global.offset == 56 and P.n_positions_global.offset == 64
    assert ctypes.sizeof(P) == 72
    assert S.full_windows.offset == 60 and S.global_counts.offset == 64 and S.n_windows_global.offset == 72
    assert ctypes.sizeof(S) == 88


def test_global_counts_need_both():
    import torch
    d = torch.empty(2, 3, 8, dtype=torch.bfloat16)
    p = aal.loss_problem(d, aal.AAL_BOTH, n_windows_global=10, n_positions_global=30)
    assert (p.global_counts, p.n_windows_global, p.n_positions_global) == (1, 10, 30)
    assert aal.loss_problem(d, aal.AAL_BOTH).global_counts == 0
    with pytest.raises(ValueError):
        aal.loss_problem(d, aal.AAL_BOTH, n_windows_global=10)
    s = aal.seq_problem(d, 2, aal.AAL_KL | aal.AAL_GREEDY, n_windows_global=6, n_positions_global=6)
    assert (s.global_counts, s.n_windows_global, s.n_positions_global) == (1, 6, 6)
