"""The one-call forward + backward of the sequence layout (aal_seq_loss_fwd_bwd).

Sec. 3.3: a window starts at every position, so a position's gradient needs the acceptances of the
K - 1 positions on each side.  The call must give the loss, the per-window expected lengths and the
gradient of aal_seq_loss_fwd followed by aal_seq_loss_bwd bit for bit: on the fused path (bf16 rows
of 16-byte multiples; every flag combination it instantiates; masks with holes, prompts and padding;
full_windows; sequences shorter than the window; fewer positions than SMs, exactly one round of
rows, and several rounds, so that rows wait on neighbours taken in the same round and in the
rounds before and after; full-size rows; token ids, with the draft alone streamed) and on the
problems it hands to the two calls (fp32, unaligned rows).  Some cases are also checked against the
oracle directly, and the bounded waits are driven to a timeout without a fault.
"""

import numpy as np
import pytest
import torch

import paper_2609_24150_gb300 as aal
import synth
import oracle
from tests.parity import (GRAD_ATOL, GRAD_RTOL, LOSS_ATOL, LOSS_RTOL, SeqRun, assert_bands, check_seq_loss,
                          check_seq_positions, seq_window_counts)

pytestmark = pytest.mark.gpu

DEV = "cuda:0"

G, S, B, KL, TV, IDS = aal.AAL_GREEDY, aal.AAL_SAMPLING, aal.AAL_BOTH, aal.AAL_KL, aal.AAL_TV, aal.AAL_IDS


@pytest.fixture(autouse=True, scope="module")
def _fuse_short_rows():
    """The fused kernel on every row it takes, short rows included (the default sends rows
    shorter than 128 KB to the two calls); restored afterwards."""
    aal.aal_debug_fused_min_row_bytes(0)
    yield
    aal.aal_debug_fused_min_row_bytes(-1)


def _bits(x):
    return x.view(torch.int16) if x.element_size() == 2 else x.view(torch.int32)


def assert_same(f, s):
    assert torch.equal(_bits(f.loss), _bits(s.loss)), (f.loss.item(), s.loss.item())
    assert torch.equal(_bits(f.eal), _bits(s.eal))
    diff = _bits(f.grad) != _bits(s.grad)
    assert not diff.any(), f"{int(diff.sum())} gradient elements differ, first at {diff.nonzero()[0].tolist()}"


def _inputs(Bn, Tn, V, seed, masked=False, dtype=torch.bfloat16):
    t, d, _ = synth.make_seq_logits("seq_tiny", seed=seed, B=Bn, seq_len=Tn, V=V, dtype=dtype, masked=False)
    mask = None
    if masked:
        g = torch.Generator().manual_seed(seed + 1)
        mask = (torch.rand((Bn, Tn), generator=g) >= 0.1).to(torch.uint8)
        mask[0, : min(3, Tn)] = 0                 # a prompt
        mask[-1, Tn - min(2, Tn):] = 0            # padding at the end
        mask = mask.to(DEV)
    return t.to(DEV), d.to(DEV), mask


def _runs(t, d, m, K, mode, T, wg, ws, dloss, full=False, wkl=1.0, wtv=1.0):
    f = SeqRun(t, d, m, K, mode, T, wg, ws, dloss, full, wkl, wtv, fused=True)
    s = SeqRun(t, d, m, K, mode, T, wg, ws, dloss, full, wkl, wtv)
    return f, s


# (B, T, K, V, mode, T, wg, ws, wkl, wtv, masked, full_windows): each fused instantiation at least
# once, over shapes that take one or several rounds of rows (152 SMs: 33 < 152, 152 = one round,
# 153 and 400 two or three rounds)
CASES = [
    (3, 11, 4, 4104, B, 1.0, 0.5, 0.5, 1.0, 1.0, True, False),      # two passes, q = q~, fewer rows than SMs
    (2, 200, 7, 2000, B, 1.0, 0.5, 0.5, 1.0, 1.0, True, False),     # three rounds of rows
    (2, 200, 7, 2000, B, 1.0, 0.5, 0.5, 1.0, 1.0, True, True),      # ... with full windows only
    (7, 50, 8, 1000, S, 0.7, 0.0, 1.0, 1.0, 1.0, True, False),      # sampling only, T != 1, K = 8
    (1, 400, 5, 8192, B, 1.5, 0.5, 0.5, 1.0, 1.0, False, False),    # greedy q beside q~ at T != 1
    (1, 152, 7, 1000, G, 1.0, 1.0, 0.0, 1.0, 1.0, True, False),     # one pass; exactly one round
    (1, 153, 7, 1000, G, 1.0, 1.0, 0.0, 1.0, 1.0, False, False),    # one row in the second round
    (4, 100, 4, 3000, KL | G, 1.0, 0.1, 0.0, 1.0, 1.0, False, False),   # one pass with the anchor
    (4, 100, 4, 3000, KL, 1.0, 0.0, 0.0, 1.0, 1.0, True, False),        # the anchor alone
    (3, 120, 6, 6000, KL | B, 1.0, 0.1, 0.1, 1.0, 1.0, True, False),    # two passes with the anchor
    (3, 120, 6, 6000, KL | TV, 1.0, 0.0, 0.0, 1.0, 0.1, False, False), # TV term + anchor
    (2, 160, 3, 4096, KL | S, 0.8, 0.5, 0.5, 1.0, 1.0, True, False),    # anchor beside WTV at T != 1
    (2, 160, 5, 9000, KL | B, 1.5, 0.1, 0.5, 1.0, 1.0, False, True),    # ... and beside EAL too
    (5, 64, 1, 4096, B, 1.0, 0.5, 0.5, 1.0, 1.0, True, False),      # K = 1: no neighbours
    (4, 3, 7, 4104, B, 1.0, 0.5, 0.5, 1.0, 1.0, False, False),      # sequences shorter than the window
    (40, 5, 6, 256, B, 1.0, 0.5, 0.5, 1.0, 1.0, True, False),       # many short sequences, several rounds
    (30, 20, 3, 8, B, 1.0, 0.5, 0.5, 1.0, 1.0, True, False),        # one 16-byte vector a row
    (1, 3, 7, 4104, B, 1.0, 0.5, 0.5, 1.0, 1.0, False, False),      # fewer rows than the window (one round)
    (64, 1, 8, 2000, B, 1.0, 0.5, 0.5, 1.0, 1.0, True, False),      # sequences of one position
]


@pytest.mark.parametrize("Bn,Tn,K,V,mode,T,wg,ws,wkl,wtv,masked,full", CASES)
@pytest.mark.parametrize("dloss_is_w", [False, True])
def test_seq_fused_equals_two_calls(Bn, Tn, K, V, mode, T, wg, ws, wkl, wtv, masked, full, dloss_is_w):
    t, d, m = _inputs(Bn, Tn, V, seed=Bn * Tn + K + V, masked=masked)
    dloss = float(seq_window_counts(m, Bn, Tn)) if dloss_is_w else 1.0
    f, s = _runs(t, d, m, K, mode, T, wg, ws, dloss, full, wkl, wtv)
    assert_same(f, s)


def test_seq_fused_workspace_serves_the_backward():
    """The workspace after the one call is the forward's: aal_seq_loss_bwd with another dloss gives
    the two calls' gradient for that dloss."""
    t, d, m = _inputs(2, 200, 2000, seed=41, masked=True)
    f = SeqRun(t, d, m, 7, B, 1.0, 0.5, 0.5, 1.0, fused=True)
    g = torch.full_like(d, float("nan"))
    aal.aal_seq_loss_bwd(f.prob, d, t, m, f.ws_buf, 3.0, g)
    s = SeqRun(t, d, m, 7, B, 1.0, 0.5, 0.5, 3.0)
    assert torch.equal(_bits(g), _bits(s.grad))


def test_seq_fused_no_valid_window():
    t, d, _ = _inputs(2, 40, 4096, seed=5)
    m = torch.zeros((2, 40), dtype=torch.uint8, device=DEV)
    f, s = _runs(t, d, m, 4, B, 1.0, 0.5, 0.5, 1.0)
    assert f.loss.item() == 0.0 and not f.grad.float().abs().gt(0).any()
    assert_same(f, s)


def test_seq_fused_empty_batch():
    d = torch.empty((0, 16, 4096), dtype=torch.bfloat16, device=DEV)
    prob = aal.seq_problem(d, 4, B, 1.0, 0.5, 0.5)
    ws = torch.empty(max(1, aal.aal_seq_workspace_size(prob)), dtype=torch.uint8, device=DEV)
    loss = torch.full((1,), float("nan"), device=DEV)
    aal.aal_seq_loss_fwd_bwd(prob, d, d, None, ws, 1.0, loss, torch.empty_like(d))
    assert loss.item() == 0.0


@pytest.mark.parametrize("mode,T,dtype,V", [
    (B, 1.0, torch.float32, 4096),        # fp32 logits
    (B, 1.0, torch.bfloat16, 1001),       # rows that are not 16-byte multiples
    (KL | S, 0.8, torch.float32, 4096),   # the anchor beside the sampling term at T != 1, fp32
])
def test_seq_problems_the_two_calls_take(mode, T, dtype, V):
    t, d, m = _inputs(3, 60, V, seed=V, masked=True, dtype=dtype)
    f, s = _runs(t, d, m, 5, mode, T, 0.5, 0.5, 1.0)
    assert_same(f, s)


@pytest.mark.parametrize("Bn,Tn,K,V,masked,full", [
    (2, 90, 4, 4096, True, False),      # fewer rows than SMs
    (2, 200, 7, 2000, True, False),     # three rounds of rows
    (2, 200, 7, 2000, True, True),      # ... full windows only
    (1, 153, 8, 1000, False, False),    # one row in the second round, K = 8
    (5, 64, 1, 4096, True, False),      # K = 1
    (4, 3, 7, 4104, False, False),      # sequences shorter than the window
    (30, 20, 3, 8, True, False),        # one 16-byte vector a row
])
@pytest.mark.parametrize("dloss_is_w", [False, True])
def test_seq_token_ids_fused_equals_two_calls(Bn, Tn, K, V, masked, full, dloss_is_w):
    """x* as token ids (AAL_GREEDY | AAL_IDS): the draft alone streamed, bitwise the two calls."""
    t, d, m = _inputs(Bn, Tn, V, seed=Bn + Tn + K + V, masked=masked)
    ids = t.float().argmax(-1).to(torch.int32).contiguous()
    dloss = float(seq_window_counts(m, Bn, Tn)) if dloss_is_w else 1.0
    f, s = _runs(ids, d, m, K, G | IDS, 1.0, 1.0, 0.0, dloss, full)
    assert_same(f, s)


def test_seq_token_ids_fused_against_the_oracle():
    """400 rows (three rounds), masked, K = 7: every output on every position against the oracle."""
    t, d, m = _inputs(2, 200, 3000, seed=37, masked=True)
    ids = t.float().argmax(-1).to(torch.int32).contiguous()
    dloss = float(seq_window_counts(m, 2, 200))
    run = SeqRun(ids, d, m, 7, G | IDS, 1.0, 1.0, 0.0, dloss, fused=True)
    ids_h, m_h = ids.cpu().numpy(), m.cpu().numpy()
    fw = oracle.seq_loss_forward(None, d.cpu(), m_h, 7, oracle.MODE_GREEDY, xstar=ids_h)
    np.testing.assert_allclose(run.eal.cpu().numpy()[:, 0], fw["eal_g"], rtol=LOSS_RTOL, atol=LOSS_ATOL)
    assert abs(run.loss.item() - fw["loss"]) <= LOSS_RTOL * abs(fw["loss"]) + LOSS_ATOL
    g_ref = oracle.seq_loss_backward(None, d.cpu(), m_h, 7, oracle.MODE_GREEDY, dloss=dloss, xstar=ids_h)
    g = run.grad.double().cpu().numpy()
    bad = np.abs(g - g_ref) > GRAD_ATOL + GRAD_RTOL * np.abs(g_ref)
    assert not bad.any(), (int(bad.sum()), tuple(np.argwhere(bad)[0]))


def test_seq_token_ids_out_of_range_reported():
    t, d, _ = _inputs(2, 100, 4096, seed=43)
    ids = t.float().argmax(-1).to(torch.int32).contiguous()
    ids[1, 17] = 4096                                   # one id past the vocabulary
    prob = aal.seq_problem(d, 5, G | IDS, 1.0, 1.0, 0.0)
    ws = torch.empty(aal.aal_seq_workspace_size(prob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    grad = torch.empty_like(d)
    aal.aal_seq_loss_fwd_bwd(prob, d, ids, None, ws, 1.0, loss, grad)
    assert aal.aal_check_device_status(ws) == aal.AAL_ERR_INVALID_ARG
    ws2 = torch.empty_like(ws)
    g2 = torch.empty_like(grad)
    aal.aal_seq_loss_fwd(prob, d, ids, None, ws2, loss)
    aal.aal_seq_loss_bwd(prob, d, ids, None, ws2, 1.0, g2)
    assert aal.aal_check_device_status(ws2) == aal.AAL_ERR_INVALID_ARG
    assert torch.equal(_bits(grad), _bits(g2))


def test_seq_token_ids_ring_times_out_and_context_stays_usable():
    t, d, _ = _inputs(2, 200, 40000, seed=12)
    ids = t.float().argmax(-1).to(torch.int32).contiguous()
    prob = aal.seq_problem(d, 7, G | IDS, 1.0, 1.0, 0.0)
    ws = torch.empty(aal.aal_seq_workspace_size(prob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    grad = torch.empty_like(d)
    aal.aal_debug_fail_next_forward(2, 50_000_000)
    try:
        aal.aal_seq_loss_fwd_bwd(prob, d, ids, None, ws, 1.0, loss, grad)
        assert aal.aal_check_device_status(ws) == aal.AAL_ERR_TIMEOUT
        assert aal.aal_check_device_status(ws) == aal.AAL_OK
    finally:
        aal.aal_debug_fail_next_forward(-1, 0)
    f, s = _runs(ids, d, None, 7, G | IDS, 1.0, 1.0, 0.0, 1.0)
    assert_same(f, s)


def test_seq_grpo_is_refused():
    t, d, _ = _inputs(1, 8, 1024, seed=1)
    with pytest.raises(aal.AalError):
        SeqRun(t, d, None, 2, G | aal.AAL_GRPO, 1.0, 1.0, 0.0, fused=True)


@pytest.mark.parametrize("mode,T,wg,ws,full", [(B, 1.0, 0.5, 0.5, False), (B, 1.3, 0.4, 0.6, True),
                                               (KL | G, 1.0, 0.1, 0.0, False), (KL | TV, 1.0, 0.0, 0.0, False)])
def test_seq_fused_against_the_oracle(mode, T, wg, ws, full):
    """B = 2 sequences of 200 positions, K = 7, V = 3000 (400 rows: three rounds on 152 SMs, rows
    whose neighbours are taken in the round before or after), masked: every output on every
    position against the oracle."""
    t, d, m = _inputs(2, 200, 3000, seed=29, masked=True)
    dloss = float(seq_window_counts(m, 2, 200))
    run = SeqRun(t, d, m, 7, mode, T, wg, ws, dloss, full, 1.0, 0.1, fused=True)
    check_seq_loss(run, t, d, m, 7, mode, T, wg, ws, dloss=dloss, full_windows=full, wkl=1.0, wtv=0.1)


def test_seq_ring_and_exchange_time_out_and_context_stays_usable():
    """One ring copy of every CTA is left unarmed: its waits run out (50 ms), the CTAs that gave
    up still publish their rows' mailbox words, and the call returns with AAL_ERR_TIMEOUT
    recorded; the next call is exact again."""
    t, d, _ = _inputs(2, 200, 20000, seed=11)
    prob = aal.seq_problem(d, 7, B, 1.0, 0.5, 0.5)
    ws = torch.empty(aal.aal_seq_workspace_size(prob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    grad = torch.empty_like(d)
    aal.aal_debug_fail_next_forward(3, 50_000_000)
    try:
        aal.aal_seq_loss_fwd_bwd(prob, d, t, None, ws, 1.0, loss, grad)
        assert aal.aal_check_device_status(ws) == aal.AAL_ERR_TIMEOUT
        assert aal.aal_check_device_status(ws) == aal.AAL_OK
    finally:
        aal.aal_debug_fail_next_forward(-1, 0)
    f, s = _runs(t, d, None, 7, B, 1.0, 0.5, 0.5, 1.0)
    assert_same(f, s)


# ------------------------------------------------------------------ full size

@pytest.fixture(scope="module")
def seq_v128k():
    return [None if x is None else x.to(DEV) for x in synth.make_seq_logits("seq_v128k", seed=0)]


def test_seq_v128k_full_size_fused_equals_two_calls(seq_v128k):
    """B = 4 x 2048 positions, K = 7, V = 128256 bf16 with prompt and padding masks (54 rounds of
    rows on 152 SMs): EAL + WTV at T = 1 and L_KL + 0.1 L_EAL, bitwise."""
    target, draft, mask = seq_v128k
    Bn, Tn, _ = draft.shape
    dloss = float(seq_window_counts(mask, Bn, Tn))
    for mode, wg, ws in [(B, 0.5, 0.5), (KL | G, 0.1, 0.0)]:
        f, s = _runs(target, draft, mask, 7, mode, 1.0, wg, ws, dloss)
        assert_same(f, s)
        del f, s


def test_seq_v128k_fused_sampled_positions(seq_v128k):
    """The fused call at full size against the oracle on sampled positions (sequence ends, both
    sides of each mask boundary, positions at the edges of a round of rows, random interior
    positions), with the batch's |W|."""
    target, draft, mask = seq_v128k
    K = 7
    Bn, Tn, _ = draft.shape
    nvalid = seq_window_counts(mask, Bn, Tn)
    dloss = float(nvalid)
    run = SeqRun(target, draft, mask, K, B, 1.0, 0.5, 0.5, dloss=dloss, fused=True)
    m = mask.cpu().numpy()
    rng = np.random.default_rng(1)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    positions = []
    for b in range(Bn):
        valid = np.flatnonzero(m[b])
        first, last = int(valid[0]), int(valid[-1])
        positions += [(b, 0), (b, first - 1), (b, first), (b, last), (b, min(Tn - 1, last + 1)),
                      (b, Tn - 1), (b, int(rng.integers(first, last + 1)))]
    # rows at the edges of a round (CTAs walk R-1-c, R-1-c-C, ...: rows R-1-i*C-c with c near 0 or C-1)
    R = Bn * Tn
    for r in (R - 1 - 5 * sms, R - 9 * sms + 2, R - 1 - 20 * sms - (sms - K + 1), R - 20 * sms):
        positions.append((r // Tn, r % Tn))
    positions = sorted({(b, t) for b, t in positions if 0 <= t < Tn})
    check_seq_positions(run, target, draft, mask, K, B, 1.0, 0.5, 0.5, dloss, positions, nvalid)
    assert_bands()
    dead = torch.from_numpy(m == 0).to(DEV)
    assert torch.count_nonzero(run.grad[dead]).item() == 0
