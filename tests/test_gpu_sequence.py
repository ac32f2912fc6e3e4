"""GPU parity of the sequence (sliding-window) layout against the fp64 oracle, through the C ABI.

Sec. 3.3: logits are stored once per position and a window of K positions starts at every
position; a position is depth j of up to K windows, and its gradient row is the sum over them.
"""

import numpy as np
import pytest
import torch

import paper_2609_24150_gb300 as aal
import synth
from tests.parity import (LOSS_ATOL, LOSS_RTOL, LossRun, SeqRun, assert_bands, check_seq_loss, check_seq_positions,
                          seq_window_counts)

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _dev(*ts):
    return [None if t is None else t.to(DEV) for t in ts]


# ------------------------------------------------------------------ small cases, every position

@pytest.mark.parametrize("mode,T,wg,ws", [
    (aal.AAL_GREEDY, 0.0, 1.0, 0.0),
    (aal.AAL_SAMPLING, 1.0, 0.0, 1.0),
    (aal.AAL_BOTH, 1.0, 0.5, 0.5),
    (aal.AAL_BOTH, 0.7, 0.3, 0.7),
])
@pytest.mark.parametrize("masked", [False, True])
def test_tiny_sequences_all_positions(mode, T, wg, ws, masked):
    target, draft, mask = synth.make_seq_logits("seq_tiny", seed=3, masked=masked)
    t, d, m = _dev(target, draft, mask)
    dloss = float(seq_window_counts(m, *d.shape[:2]))   # gradients O(q): the absolute tolerance binds
    run = SeqRun(t, d, m, 4, mode, T, wg, ws, dloss=dloss)
    check_seq_loss(run, t, d, m, 4, mode, T, wg, ws, dloss=dloss)


@pytest.mark.parametrize("V,dtype", [(7, torch.bfloat16), (4099, torch.float32), (4104, torch.bfloat16),
                                     (65544, torch.bfloat16)])
@pytest.mark.parametrize("K", [1, 3, 8])
def test_ragged_vocab_and_window_sizes(V, dtype, K):
    """Generic and streamed row kernels (V*elem a multiple of 16 bytes or not), K from 1 to 8,
    a sequence shorter than the window, and a hole in the middle of a sequence."""
    B, Tn = 3, 11
    target, draft, _ = synth.make_seq_logits("seq_tiny", seed=V + K, B=B, seq_len=Tn, V=V, dtype=dtype,
                                             masked=False)
    mask = torch.ones(B, Tn, dtype=torch.uint8)
    mask[1, 4] = 0
    mask[2, :2] = 0
    mask[2, 9:] = 0
    t, d, m = _dev(target, draft, mask)
    dloss = float(seq_window_counts(m, B, Tn))
    for mode, T in [(aal.AAL_BOTH, 1.0), (aal.AAL_BOTH, 1.3), (aal.AAL_GREEDY, 0.0)]:
        run = SeqRun(t, d, m, K, mode, T, 0.5, 0.5, dloss=dloss)
        check_seq_loss(run, t, d, m, K, mode, T, 0.5, 0.5, dloss=dloss)
    # sequences shorter than the window
    ts, ds = t[:, :2].contiguous(), d[:, :2].contiguous()
    run = SeqRun(ts, ds, None, K, aal.AAL_BOTH, 1.0, 0.5, 0.5, dloss=2.0 * B)
    check_seq_loss(run, ts, ds, None, K, aal.AAL_BOTH, 1.0, 0.5, 0.5, dloss=2.0 * B)


def test_long_sequence_spans_many_window_blocks():
    """3000 windows: several window-kernel blocks, the last-block loss reduction, and gathers
    that read partials written by neighbouring blocks."""
    target, draft, _ = synth.make_seq_logits("seq_tiny", seed=11, B=1, seq_len=3000, V=64, masked=False)
    mask = torch.ones(1, 3000, dtype=torch.uint8)
    mask[0, 255:258] = 0            # holes at a window-block boundary
    mask[0, 1023] = 0
    t, d, m = _dev(target, draft, mask)
    run = SeqRun(t, d, m, 8, aal.AAL_BOTH, 0.9, 0.4, 0.6, dloss=2996.0)
    check_seq_loss(run, t, d, m, 8, aal.AAL_BOTH, 0.9, 0.4, 0.6, dloss=2996.0)


# ------------------------------------------------------------------ agreement with the windowed path

def _gather_on_device(target, draft, mask, K):
    """Windows [B*T][K][V] gathered by indexing (test plumbing), with their validity."""
    B, Tn, V = draft.shape
    t = torch.arange(Tn, device=draft.device)
    j = torch.arange(K, device=draft.device)
    pos = t[:, None] + j[None, :]                                  # [T][K]
    inside = pos < Tn
    pos = pos.clamp(max=Tn - 1)
    wp = target[:, pos].reshape(B * Tn, K, V).contiguous()
    wq = draft[:, pos].reshape(B * Tn, K, V).contiguous()
    valid = inside[None].expand(B, Tn, K)
    if mask is not None:
        valid = valid & (mask[:, pos] != 0)
    return wp, wq, valid.reshape(B * Tn, K).to(torch.uint8).contiguous(), pos, inside


@pytest.mark.parametrize("mode,T", [(aal.AAL_BOTH, 1.0), (aal.AAL_SAMPLING, 0.8), (aal.AAL_GREEDY, 0.0)])
def test_same_windows_as_the_windowed_layout(mode, T):
    """Gathering the windows and running the windowed entry points gives bit-identical per-window
    expected lengths and loss (same row statistics, same window arithmetic, same reduction
    order); the gradient rows scatter-added back agree to fp32 rounding."""
    target, draft, mask = synth.make_seq_logits("seq_tiny", seed=5, B=2, seq_len=300, V=2048)
    t, d, m = _dev(target, draft, mask)
    K = 5
    seq = SeqRun(t, d, m, K, mode, T, 0.3, 0.7, dloss=7.0)
    wp, wq, wm, pos, inside = _gather_on_device(t, d, m, K)
    win = LossRun(wp, wq, wm, mode, T, 0.3, 0.7, dloss=7.0)
    assert torch.equal(seq.eal, win.eal)
    assert torch.equal(seq.loss, win.loss)
    B, Tn, V = d.shape
    g = torch.zeros(B, Tn, V, dtype=torch.float64, device=DEV)
    wg = win.grad.double().view(B, Tn, K, V)
    for j in range(K):
        ok = inside[:, j]
        g[:, pos[ok, j]] += wg[:, ok, j]
    np.testing.assert_allclose(seq.grad.double().cpu().numpy(), g.cpu().numpy(), rtol=1e-4, atol=1e-9)


# ------------------------------------------------------------------ edge cases

def test_empty_batch_and_empty_sequences():
    for B, Tn in [(0, 16), (3, 0)]:
        d = torch.zeros(B, Tn, 64, dtype=torch.bfloat16, device=DEV)
        prob = aal.seq_problem(d, 4, aal.AAL_BOTH)
        ws = torch.empty(max(1, aal.aal_seq_workspace_size(prob)), dtype=torch.uint8, device=DEV)
        loss = torch.full((1,), float("nan"), device=DEV)
        aal.aal_seq_loss_fwd(prob, d, d, None, ws, loss)
        aal.aal_seq_loss_bwd(prob, d, d, None, ws, 1.0, d)
        torch.cuda.synchronize()
        assert loss.item() == 0.0


def test_all_positions_masked():
    target, draft, _ = synth.make_seq_logits("seq_tiny", seed=2, B=2, seq_len=9, V=512,
                                             dtype=torch.bfloat16, masked=False)
    t, d = _dev(target, draft)
    m = torch.zeros(2, 9, dtype=torch.uint8, device=DEV)
    run = SeqRun(t, d, m, 4, aal.AAL_BOTH, 1.0, 0.5, 0.5)
    assert run.loss.item() == 0.0
    assert torch.count_nonzero(run.grad).item() == 0
    assert torch.count_nonzero(run.eal).item() == 0


def test_identical_draft_and_target():
    """q = p: every sampling acceptance is 1, so E^s = K_n and the WTV gradient is zero; the
    greedy gradient is not (a^g = q(x*) < 1)."""
    target, _, mask = synth.make_seq_logits("seq_tiny", seed=4, V=3000, dtype=torch.bfloat16)
    t, m = _dev(target, mask)
    K = 4
    run = SeqRun(t, t, m, K, aal.AAL_SAMPLING, 1.0, 0.0, 1.0)
    B, Tn = m.shape
    kn = torch.zeros(B, Tn, device=DEV)
    for b in range(B):
        for s in range(Tn):
            k = 0
            while k < K and s + k < Tn and m[b, s + k] != 0:
                k += 1
            kn[b, s] = k
    np.testing.assert_allclose(run.eal[:, 1].cpu().numpy(), kn.flatten().cpu().numpy(), rtol=1e-5, atol=0)
    assert torch.count_nonzero(run.grad).item() == 0


# ------------------------------------------------------------------ full size, sampled positions

@pytest.fixture(scope="module")
def seq_v128k():
    return _dev(*synth.make_seq_logits("seq_v128k", seed=0))


@pytest.mark.parametrize("mode,T,wg,ws", [(aal.AAL_BOTH, 1.0, 0.5, 0.5), (aal.AAL_SAMPLING, 0.8, 0.0, 1.0)])
def test_full_size_sampled_positions(seq_v128k, mode, T, wg, ws):
    """B=4 x 2048 positions, K=7, V=128256 bf16 with prompt and padding masks: the window
    starting at, and the gradient row of, sampled positions (sequence ends, both sides of each
    mask boundary, and random interior positions) against the oracle; the loss against the
    per-window outputs, and all gradient rows outside every valid window exactly zero."""
    target, draft, mask = seq_v128k
    K = 7
    B, Tn, V = draft.shape
    dloss = float(seq_window_counts(mask, B, Tn))    # gradients O(q): the absolute tolerance binds
    run = SeqRun(target, draft, mask, K, mode, T, wg, ws, dloss=dloss)
    nvalid = seq_window_counts(mask, B, Tn)
    m = mask.cpu().numpy()
    rng = np.random.default_rng(0)
    positions = []
    for b in range(B):
        valid = np.flatnonzero(m[b])
        first, last = int(valid[0]), int(valid[-1])
        positions += [(b, 0), (b, first - 1), (b, first), (b, last), (b, min(Tn - 1, last + 1)),
                      (b, Tn - 1), (b, int(rng.integers(first, last + 1)))]
    positions = sorted({(b, t) for b, t in positions if 0 <= t < Tn})
    check_seq_positions(run, target, draft, mask, K, mode, T, wg, ws, dloss, positions, nvalid)
    assert_bands()
    eal = run.eal.double().cpu().numpy()
    num = (wg * eal[:, 0].sum() if mode & aal.AAL_GREEDY else 0.0) + \
          (ws * eal[:, 1].sum() if mode & aal.AAL_SAMPLING else 0.0)
    ref = -num / nvalid
    assert abs(run.loss.item() - ref) <= LOSS_RTOL * abs(ref) + LOSS_ATOL
    # a position belongs to some valid window prefix iff it is valid itself
    dead = torch.from_numpy(m == 0).to(DEV)
    assert torch.count_nonzero(run.grad[dead]).item() == 0
    assert torch.count_nonzero(run.eal.view(B, Tn, 2)[dead]).item() == 0


@pytest.mark.parametrize("K", [1, 4, 8])
def test_full_windows_reading(K):
    """full_windows = 1: only windows whose K positions are all valid count (and get gradient)."""
    target, draft, mask = synth.make_seq_logits("seq_tiny", seed=8 + K)
    t, d, m = _dev(target, draft, mask)
    for mm in (None, m):
        kn_full = SeqRun(t, d, mm, K, aal.AAL_BOTH, 1.0, 0.5, 0.5, full_windows=True)
        dloss = float(max(1, torch.count_nonzero(kn_full.eal[:, 0]).item()))
        run = SeqRun(t, d, mm, K, aal.AAL_BOTH, 1.0, 0.5, 0.5, dloss=dloss, full_windows=True)
        check_seq_loss(run, t, d, mm, K, aal.AAL_BOTH, 1.0, 0.5, 0.5, dloss=dloss, full_windows=True)
