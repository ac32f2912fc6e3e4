"""GPU parity of the forward-KL anchor (mode bit AAL_KL, Sec. 4.1) against the fp64 oracle,
in both layouts, through the C ABI.  The greedy-regime objective of the paper is
L_KL + 0.1 L_EAL: mode AAL_KL | AAL_GREEDY with w_kl = 1, w_greedy = 0.1."""

import numpy as np
import pytest
import torch

import oracle
import paper_2609_24150_gb300 as aal
import synth
from tests.parity import (LossRun, SeqRun, assert_bands, check_loss, check_seq_loss, check_seq_positions,
                          seq_window_counts)

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
KL_G = aal.AAL_KL | aal.AAL_GREEDY


def _dev(*ts):
    return [None if t is None else t.to(DEV) for t in ts]


def _npos(mask, n):
    return n if mask is None else int((mask != 0).sum().item())


@pytest.mark.parametrize("mode,T,wg,ws,wkl", [
    (KL_G, 0.0, 0.1, 0.0, 1.0),                         # the paper's greedy-regime objective
    (aal.AAL_KL, 0.0, 0.0, 0.0, 1.0),                   # the L_KL baseline
    (aal.AAL_KL | aal.AAL_SAMPLING, 0.8, 0.0, 1.0, 0.5),
    (aal.AAL_KL | aal.AAL_BOTH, 1.0, 0.3, 0.7, 2.0),    # T = 1: q = q~ shared by three terms
])
@pytest.mark.parametrize("masked", [False, True])
def test_tiny_all_rows(mode, T, wg, ws, wkl, masked):
    target, draft, _ = synth.make_logits("tiny", seed=21)
    mask = None
    if masked:
        mask = torch.ones(32, 4, dtype=torch.uint8)
        mask[3, 0] = 0          # window leaves W, its later positions stay valid for the anchor
        mask[5, 2:] = 0
        mask[9, :] = 0
    t, d, m = _dev(target, draft, mask)
    dloss = float(_npos(mask, 32 * 4))
    run = LossRun(t, d, m, mode, T, wg, ws, dloss=dloss, wkl=wkl)
    check_loss(run, t, d, m, mode, T, wg, ws, dloss=dloss, wkl=wkl)


@pytest.mark.parametrize("V,dtype", [(7, torch.bfloat16), (4099, torch.float32), (4104, torch.bfloat16)])
@pytest.mark.parametrize("K", [1, 3])
def test_ragged_vocab(V, dtype, K):
    target, draft, _ = synth.make_logits("tiny", seed=V + 3 * K, N=6, K=K, V=V, dtype=dtype)
    t, d = _dev(target, draft)
    for mode, T in [(KL_G, 0.0), (aal.AAL_KL | aal.AAL_BOTH, 1.3)]:
        run = LossRun(t, d, None, mode, T, 0.1, 0.5, dloss=6.0 * K, wkl=1.0)
        check_loss(run, t, d, None, mode, T, 0.1, 0.5, dloss=6.0 * K, wkl=1.0)


def test_full_vocabulary_rows():
    """V = 128256 bf16 rows of the bench workload, every row (the per-row arithmetic does
    not depend on how many rows a launch holds)."""
    target, draft, _ = synth.make_logits("v128k", seed=0, n_windows=8)
    t, d = _dev(target, draft)
    dloss = 8.0 * 7
    run = LossRun(t, d, None, KL_G, 0.0, 0.1, 0.0, dloss=dloss, wkl=1.0)
    check_loss(run, t, d, None, KL_G, 0.0, 0.1, 0.0, dloss=dloss, wkl=1.0)


def test_identical_rows_have_zero_kl():
    target, _, _ = synth.make_logits("v152k", seed=5, N=4, K=3, V=4000)
    t = target.to(DEV)
    run = LossRun(t, t.clone(), None, aal.AAL_KL, 0.0, 0.0, 0.0, dloss=12.0)
    assert abs(run.loss.item()) < 1e-6
    assert float(run.grad.float().abs().max()) < 1e-5


def test_anchor_adds_to_the_window_terms():
    """The loss of KL | GREEDY is the loss of GREEDY plus w_kl times the loss of KL alone."""
    target, draft, mask = synth.make_logits("v32k", seed=2, n_windows=64)
    t, d, m = _dev(target, draft, mask)
    a = LossRun(t, d, m, KL_G, 0.0, 0.1, 0.0, wkl=0.7).loss.item()
    b = LossRun(t, d, m, aal.AAL_GREEDY, 0.0, 0.1, 0.0).loss.item()
    c = LossRun(t, d, m, aal.AAL_KL, 0.0, 0.0, 0.0, wkl=1.0).loss.item()
    assert abs(a - (b + 0.7 * c)) <= 1e-5 * (abs(a) + 1e-3)
    assert c > 0


def test_full_size_sampled_windows_greedy_objective():
    """N = 8192 windows, K = 7, V = 128256 bf16 under L_KL + 0.1 L_EAL: sampled windows'
    gradient rows and expected lengths against the oracle with the batch's |W| and |P|."""
    target, draft, _ = synth.make_logits("v128k", seed=0, device=DEV)
    N, K, V = draft.shape
    run = LossRun(target, draft, None, KL_G, 0.0, 0.1, 0.0, dloss=float(N * K), wkl=1.0)
    windows = [0, 1, 4095, 8191]
    check_loss(run, target, draft, None, KL_G, 0.0, 0.1, 0.0, dloss=float(N * K), windows=windows,
               n_windows_total=N, wkl=1.0, n_positions_total=N * K)
    assert_bands()
    assert np.isfinite(run.loss.item())


# ------------------------------------------------------------------ sequence layout

@pytest.mark.parametrize("mode,T,wg,ws", [(KL_G, 0.0, 0.1, 0.0), (aal.AAL_KL | aal.AAL_SAMPLING, 0.9, 0.0, 1.0)])
@pytest.mark.parametrize("full_windows", [False, True])
def test_sequence_layout(mode, T, wg, ws, full_windows):
    target, draft, mask = synth.make_seq_logits("seq_tiny", seed=13)
    t, d, m = _dev(target, draft, mask)
    dloss = float(_npos(m, 3 * 37))
    run = SeqRun(t, d, m, 4, mode, T, wg, ws, dloss=dloss, full_windows=full_windows, wkl=1.0)
    check_seq_loss(run, t, d, m, 4, mode, T, wg, ws, dloss=dloss, full_windows=full_windows, wkl=1.0)


def test_sequence_full_size_sampled_positions():
    target, draft, mask = _dev(*synth.make_seq_logits("seq_v128k", seed=1))
    B, Tn, V = draft.shape
    K = 7
    npos = _npos(mask, B * Tn)
    run = SeqRun(target, draft, mask, K, KL_G, 0.0, 0.1, 0.0, dloss=float(npos), wkl=1.0)
    m = mask.cpu().numpy()
    positions = []
    for b in range(B):
        valid = np.flatnonzero(m[b])
        positions += [(b, int(valid[0])), (b, int(valid[-1])), (b, int(valid[len(valid) // 2]))]
    check_seq_positions(run, target, draft, mask, K, KL_G, 0.0, 0.1, 0.0, float(npos), positions,
                        seq_window_counts(mask, B, Tn), wkl=1.0, npos_total=npos)
    assert_bands()
    dead = torch.from_numpy(m == 0).to(DEV)
    assert torch.count_nonzero(run.grad[dead]).item() == 0


# ------------------------------------------------------------------ the L_TV baseline term (AAL_TV)

KL_TV = aal.AAL_KL | aal.AAL_TV


@pytest.mark.parametrize("mode,T,wtv", [
    (KL_TV, 1.0, 0.1),                                # the paper's L_KL + 0.1 L_TV baseline, T = 1
    (KL_TV, 0.7, 0.1),                                # ... at T = 0.7 (z_p kept at T = 1 beside T)
    (aal.AAL_TV, 1.3, 1.0),                           # the TV term alone
    (aal.AAL_TV | aal.AAL_BOTH, 1.0, 0.5),            # beside EAL and WTV: one sampling coefficient
])
@pytest.mark.parametrize("masked", [False, True])
def test_tv_term_tiny_all_rows(mode, T, wtv, masked):
    target, draft, _ = synth.make_logits("tiny", seed=31)
    mask = None
    if masked:
        mask = torch.ones(32, 4, dtype=torch.uint8)
        mask[2, 1] = 0
        mask[6, 0] = 0
        mask[7, 3] = 0
    t, d, m = _dev(target, draft, mask)
    dloss = 32.0 * 4
    run = LossRun(t, d, m, mode, T, 0.3, 0.6, dloss=dloss, wkl=1.0, wtv=wtv)
    check_loss(run, t, d, m, mode, T, 0.3, 0.6, dloss=dloss, wkl=1.0, wtv=wtv)


@pytest.mark.parametrize("V,dtype", [(4104, torch.bfloat16), (4099, torch.float32)])
def test_tv_term_sequence_layout(V, dtype):
    target, draft, _ = synth.make_seq_logits("seq_tiny", seed=17, B=2, seq_len=13, V=V, dtype=dtype, masked=False)
    mask = torch.ones(2, 13, dtype=torch.uint8)
    mask[1, 9:] = 0
    t, d, m = _dev(target, draft, mask)
    for full in (False, True):
        run = SeqRun(t, d, m, 4, KL_TV, 0.9, 0.0, 0.0, dloss=24.0, full_windows=full, wkl=1.0, wtv=0.1)
        check_seq_loss(run, t, d, m, 4, KL_TV, 0.9, 0.0, 0.0, dloss=24.0, full_windows=full, wkl=1.0, wtv=0.1)


def test_tv_baseline_full_size_sampled_windows():
    """N = 8192 windows, K = 7, V = 128256 bf16 under L_KL + 0.1 L_TV at T = 1."""
    target, draft, _ = synth.make_logits("v128k", seed=2, device=DEV)
    N, K, V = draft.shape
    run = LossRun(target, draft, None, KL_TV, 1.0, 0.0, 0.0, dloss=float(N * K), wkl=1.0, wtv=0.1)
    check_loss(run, target, draft, None, KL_TV, 1.0, 0.0, 0.0, dloss=float(N * K), windows=[0, 3000, 8191],
               n_windows_total=N, wkl=1.0, n_positions_total=N * K, wtv=0.1)
    assert_bands()
