"""The one-call forward + backward (aal_loss_fwd_bwd).

It must give the loss, the per-window expected lengths and the gradient of aal_loss_fwd followed
by aal_loss_bwd bit for bit: on the fused path (bf16 rows of 16-byte multiples; every flag
combination it instantiates, masks, fewer windows than CTA groups, K = 1 and K = 8, windows
enough for the solo CTAs, full-size rows; token ids with the draft alone streamed) and on the problems it hands to the two calls
(fp32, unaligned rows).  A few cases are also checked against the oracle
directly, and the bounded waits are driven to a timeout without a fault.
"""

import pytest
import torch

import paper_2609_24150_gb300 as aal
import synth
from tests.parity import LossRun, check_loss

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(autouse=True, scope="module")
def _fuse_short_rows():
    """The fused kernels on every row they take, short rows included (the default sends rows
    shorter than 128 KB to the two calls, which are faster there); restored afterwards."""
    aal.aal_debug_fused_min_row_bytes(0)
    yield
    aal.aal_debug_fused_min_row_bytes(-1)


G, S, B, KL, TV, IDS = aal.AAL_GREEDY, aal.AAL_SAMPLING, aal.AAL_BOTH, aal.AAL_KL, aal.AAL_TV, aal.AAL_IDS


class FusedRun:
    """aal_loss_fwd_bwd of one problem; the same fields as LossRun."""

    def __init__(self, target, draft, mask, mode, T=1.0, wg=1.0, ws=1.0, dloss=1.0, wkl=1.0, wtv=1.0):
        self.prob = aal.loss_problem(draft, mode, T, wg, ws, wkl, wtv)
        self.ws_buf = torch.empty(aal.aal_workspace_size(self.prob), dtype=torch.uint8, device=draft.device)
        N = draft.shape[0]
        self.loss = torch.full((1,), float("nan"), dtype=torch.float32, device=draft.device)
        self.eal = torch.full((max(N, 1), 2), float("nan"), dtype=torch.float32, device=draft.device)
        self.grad = torch.full_like(draft, float("nan"))
        aal.aal_loss_fwd_bwd(self.prob, draft, target, mask, self.ws_buf, dloss, self.loss, self.grad,
                             self.eal if N > 0 else None)
        torch.cuda.synchronize()
        assert aal.aal_check_device_status(self.ws_buf) == aal.AAL_OK


def _bits(x):
    return x.view(torch.int16) if x.element_size() == 2 else x.view(torch.int32)


def assert_same(f, s):
    assert torch.equal(_bits(f.loss), _bits(s.loss)), (f.loss.item(), s.loss.item())
    assert torch.equal(_bits(f.eal), _bits(s.eal))
    diff = _bits(f.grad) != _bits(s.grad)
    assert not diff.any(), f"{int(diff.sum())} gradient elements differ, first at {diff.nonzero()[0].tolist()}"


def _inputs(N, K, V, seed, masked=False, dtype=torch.bfloat16):
    t, d, _ = synth.make_logits("tiny", seed=seed, N=N, K=K, V=V, dtype=dtype)
    mask = None
    if masked:
        g = torch.Generator().manual_seed(seed + 1)
        mask = (torch.rand((N, K), generator=g) >= 0.15).to(torch.uint8)
        mask[0, 0] = 0                        # a window outside W
        mask[1, :] = 1                        # a full window
        mask = mask.to(DEV)
    return t.to(DEV), d.to(DEV), mask


# (N, K, V, mode, T, wg, ws, wkl, wtv, masked): each fused instantiation at least once
CASES = [
    (24, 7, 4104, B, 1.0, 0.5, 0.5, 1.0, 1.0, False),       # two passes, q = q~ at T = 1
    (40, 5, 20000, S, 0.7, 1.0, 1.0, 1.0, 1.0, True),       # sampling only, T != 1, two chunks a row
    (16, 8, 8192, B, 1.5, 0.5, 0.5, 1.0, 1.0, False),       # greedy q beside q~ at T != 1
    (33, 3, 1000, G, 1.0, 1.0, 0.0, 1.0, 1.0, True),        # one pass, argmaxes resolved from L2
    (20, 4, 3000, KL | G, 1.0, 0.1, 0.0, 1.0, 1.0, False),  # one pass with the anchor
    (20, 4, 3000, KL, 1.0, 0.0, 0.0, 1.0, 1.0, True),       # the anchor alone
    (12, 6, 6000, KL | B, 1.0, 0.1, 0.1, 1.0, 1.0, True),   # two passes with the anchor
    (12, 6, 6000, KL | TV, 1.0, 0.0, 0.0, 1.0, 0.1, False), # TV term + anchor, no greedy term
    (10, 3, 4096, KL | S, 0.8, 0.5, 0.5, 1.0, 1.0, True),   # the anchor beside WTV at T != 1: z_p and z_q at 1 and T
    (14, 5, 9000, KL | B, 1.5, 0.1, 0.5, 1.0, 1.0, False),  # ... and beside EAL too
    (3, 7, 128256, B, 1.0, 0.5, 0.5, 1.0, 1.0, False),      # fewer windows than groups, full rows
    (200, 1, 2048, B, 1.0, 0.5, 0.5, 1.0, 1.0, False),      # K = 1: groups of one CTA
    (30, 3, 8, B, 1.0, 0.5, 0.5, 1.0, 1.0, True),           # one 16-byte vector a row
    (30, 4, 24, KL | G, 1.0, 0.1, 0.0, 1.0, 1.0, False),    # three vectors a row, one pass
]


# Windows enough that the SMs the groups leave over (152 - G K) take whole windows as solo CTAs:
# again each instantiation once.  N = G K + S balances one window per solo CTA; 304, two.
SOLO_CASES = [
    (152, 7, 4104, B, 1.0, 0.5, 0.5, 1.0, 1.0, False),
    (304, 7, 2000, S, 0.7, 1.0, 1.0, 1.0, 1.0, True),
    (152, 5, 8192, B, 1.5, 0.5, 0.5, 1.0, 1.0, False),
    (152, 3, 1000, G, 1.0, 1.0, 0.0, 1.0, 1.0, True),
    (152, 6, 3000, KL | G, 1.0, 0.1, 0.0, 1.0, 1.0, False),
    (152, 6, 3000, KL, 1.0, 0.0, 0.0, 1.0, 1.0, True),
    (152, 5, 6000, KL | B, 1.0, 0.1, 0.1, 1.0, 1.0, True),
    (152, 7, 6000, KL | TV, 1.0, 0.0, 0.0, 1.0, 0.1, False),
    (152, 5, 3000, KL | S, 0.8, 0.0, 1.0, 1.0, 1.0, True),
    (152, 6, 2000, KL | B, 1.5, 0.1, 0.5, 1.0, 1.0, False),
]


def solo_windows(N, K, sms):
    """The windows the launch gives to solo CTAs (one CTA per SM, as the ring's shared memory
    allows): the library's own split (checked against a brute force in test_abi)."""
    G = min(sms // K, N, 1024)
    S = sms - G * K
    return aal.aal_debug_solo_windows(N, K, G, S) * S if G > 0 and S > 0 else 0


@pytest.mark.parametrize("N,K,V,mode,T,wg,ws,wkl,wtv,masked", CASES + SOLO_CASES)
@pytest.mark.parametrize("dloss_is_w", [False, True])
def test_fused_equals_two_calls(N, K, V, mode, T, wg, ws, wkl, wtv, masked, dloss_is_w):
    if (N, K, V, mode, T, wg, ws, wkl, wtv, masked) in SOLO_CASES:
        sms = torch.cuda.get_device_properties(0).multi_processor_count
        assert solo_windows(N, K, sms) > 0, "the case no longer reaches the solo CTAs"
    t, d, m = _inputs(N, K, V, seed=N + K + V, masked=masked)
    dloss = float(N) if dloss_is_w else 1.0   # |W|-sized upstream gradient makes the absolute term bind
    f = FusedRun(t, d, m, mode, T, wg, ws, dloss, wkl, wtv)
    s = LossRun(t, d, m, mode, T, wg, ws, dloss, wkl, wtv)
    assert_same(f, s)


def test_fused_no_valid_window():
    t, d, _ = _inputs(8, 4, 4096, seed=5)
    m = torch.zeros((8, 4), dtype=torch.uint8, device=DEV)
    f = FusedRun(t, d, m, B, 1.0, 0.5, 0.5)
    assert f.loss.item() == 0.0 and not f.grad.float().abs().gt(0).any()
    assert_same(f, LossRun(t, d, m, B, 1.0, 0.5, 0.5))


@pytest.mark.parametrize("mode,T,dtype,V", [
    (B, 1.0, torch.float32, 4096),        # fp32 logits
    (B, 1.0, torch.bfloat16, 1001),       # rows that are not 16-byte multiples
    (KL | S, 0.8, torch.float32, 4096),   # the anchor beside the sampling term at T != 1, fp32
])
def test_problems_the_two_calls_take(mode, T, dtype, V):
    t, d, m = _inputs(10, 3, V, seed=V, masked=True, dtype=dtype)
    assert_same(FusedRun(t, d, m, mode, T, 0.5, 0.5), LossRun(t, d, m, mode, T, 0.5, 0.5))


@pytest.mark.parametrize("N,K,V,masked", [(10, 3, 4096, False), (40, 7, 30000, True), (3, 8, 128256, False),
                                           (100, 1, 1000, True), (20, 5, 8, True),
                                           (152, 7, 4096, True), (304, 5, 2000, False)])   # with solo CTAs
@pytest.mark.parametrize("dloss_is_w", [False, True])
def test_token_ids_fused_equals_two_calls(N, K, V, masked, dloss_is_w):
    """x* as token ids (the draft alone streamed), some ids out of range on one run."""
    t, d, m = _inputs(N, K, V, seed=9 + N, masked=masked)
    ids = t.float().argmax(-1).to(torch.int32).contiguous()
    dloss = float(N) if dloss_is_w else 1.0
    assert_same(FusedRun(ids, d, m, G | IDS, 1.0, 1.0, 0.0, dloss), LossRun(ids, d, m, G | IDS, 1.0, 1.0, 0.0, dloss))


def test_token_ids_out_of_range_reported():
    t, d, _ = _inputs(12, 4, 4096, seed=21)
    ids = t.float().argmax(-1).to(torch.int32).contiguous()
    ids[3, 1] = 4096                                   # one id past the vocabulary
    prob = aal.loss_problem(d, G | IDS, 1.0, 1.0, 0.0)
    ws = torch.empty(aal.aal_workspace_size(prob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    grad = torch.empty_like(d)
    aal.aal_loss_fwd_bwd(prob, d, ids, None, ws, 1.0, loss, grad)
    assert aal.aal_check_device_status(ws) == aal.AAL_ERR_INVALID_ARG
    s = torch.empty_like(grad)
    ws2 = torch.empty_like(ws)
    aal.aal_loss_fwd(prob, d, ids, None, ws2, loss)
    aal.aal_loss_bwd(prob, d, ids, None, ws2, 1.0, s)
    assert aal.aal_check_device_status(ws2) == aal.AAL_ERR_INVALID_ARG
    assert torch.equal(_bits(grad), _bits(s))


@pytest.mark.parametrize("mode,T,wg,ws", [(B, 1.0, 0.5, 0.5), (B, 1.5, 0.5, 0.5), (KL | G, 1.0, 0.1, 0.0)])
def test_fused_against_the_oracle_with_solo_ctas(mode, T, wg, ws):
    """N = 304 windows of K = 7 at V = 50000 (five ring chunks a pass, a partial last one): on
    one GB300 the call runs 21 groups of 7 CTAs with about 14 windows each and 5 solo CTAs with
    whole windows, so both paths walk several windows.  Sampled windows of each kind (every
    group's first and last window, and the solo CTAs' windows at the end of the batch) are
    checked against the oracle directly, with the batch's |W| and |P|."""
    N, K, V = 304, 7, 50000
    t, d, m = _inputs(N, K, V, seed=23, masked=True)
    run = FusedRun(t, d, m, mode, T, wg, ws, dloss=float(N), wkl=1.0)
    mh = m.cpu().numpy()
    nW = int((mh[:, 0] != 0).sum())
    nP = int((mh != 0).sum())
    groups = 21
    windows = sorted(set([0, groups - 1, groups, 2 * groups + 5] + list(range(N - 12, N)) +
                         [N - 12 - groups + 3, 150]))
    check_loss(run, t, d, m, mode, T, wg, ws, dloss=float(N), windows=windows, n_windows_total=nW, wkl=1.0,
               n_positions_total=nP)
    assert_same(run, LossRun(t, d, m, mode, T, wg, ws, dloss=float(N), wkl=1.0))


@pytest.mark.parametrize("N,K", [(16, 2), (152, 7)])   # groups only; groups and solo CTAs
def test_token_ids_ring_times_out_and_context_stays_usable(N, K):
    t, d, _ = _inputs(N, K, 40000, seed=12)
    ids = t.float().argmax(-1).to(torch.int32).contiguous()
    prob = aal.loss_problem(d, G | IDS, 1.0, 1.0, 0.0)
    ws = torch.empty(aal.aal_workspace_size(prob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    grad = torch.empty_like(d)
    aal.aal_debug_fail_next_forward(2, 50_000_000)    # a group's gradient chunk, a solo CTA's statistics chunk
    try:
        aal.aal_loss_fwd_bwd(prob, d, ids, None, ws, 1.0, loss, grad)
        assert aal.aal_check_device_status(ws) == aal.AAL_ERR_TIMEOUT
        assert aal.aal_check_device_status(ws) == aal.AAL_OK
    finally:
        aal.aal_debug_fail_next_forward(-1, 0)
    assert_same(FusedRun(ids, d, None, G | IDS, 1.0, 1.0, 0.0), LossRun(ids, d, None, G | IDS, 1.0, 1.0, 0.0))


def test_grpo_is_refused():
    t, d, _ = _inputs(4, 2, 1024, seed=1)
    with pytest.raises(aal.AalError):
        FusedRun(t, d, None, G | aal.AAL_GRPO, 1.0, 1.0, 0.0)


@pytest.mark.parametrize("mode,T,wg,ws", [(B, 1.0, 0.5, 0.5), (KL | G, 1.0, 0.1, 0.0), (S, 1.3, 0.0, 1.0),
                                         (KL | B, 0.7, 0.1, 0.5)])
def test_fused_against_the_oracle(mode, T, wg, ws):
    t, d, m = _inputs(24, 5, 3000, seed=17, masked=True)
    check_loss(FusedRun(t, d, m, mode, T, wg, ws, dloss=24.0), t, d, m, mode, T, wg, ws, dloss=24.0)


@pytest.mark.parametrize("N,K", [(16, 2), (152, 7)])   # groups only; groups and solo CTAs
def test_group_barrier_and_ring_time_out_and_context_stays_usable(N, K):
    """One ring copy of every CTA is left unarmed: its waits run out (50 ms), the CTAs that gave
    up still publish their rows' mailbox words (so no window's exchange waits the whole limit),
    and the call returns with AAL_ERR_TIMEOUT recorded."""
    t, d, _ = _inputs(N, K, 20000, seed=11)
    prob = aal.loss_problem(d, B, 1.0, 0.5, 0.5)
    ws = torch.empty(aal.aal_workspace_size(prob), dtype=torch.uint8, device=DEV)
    loss = torch.empty(1, device=DEV)
    grad = torch.empty_like(d)
    aal.aal_debug_fail_next_forward(3, 50_000_000)
    try:
        aal.aal_loss_fwd_bwd(prob, d, t, None, ws, 1.0, loss, grad)
        assert aal.aal_check_device_status(ws) == aal.AAL_ERR_TIMEOUT
        assert aal.aal_check_device_status(ws) == aal.AAL_OK
    finally:
        aal.aal_debug_fail_next_forward(-1, 0)
    assert_same(FusedRun(t, d, None, B, 1.0, 0.5, 0.5), LossRun(t, d, None, B, 1.0, 0.5, 0.5))


def test_v128k_full_size_fused_equals_two_calls():
    t, d, _ = synth.make_logits("v128k", seed=0, device=DEV)
    f = FusedRun(t, d, None, B, 1.0, 0.5, 0.5)
    s = LossRun(t, d, None, B, 1.0, 0.5, 0.5)
    assert_same(f, s)
    del f, s
    f = FusedRun(t, d, None, KL | G, 1.0, 0.1, 0.0)
    s = LossRun(t, d, None, KL | G, 1.0, 0.1, 0.0)
    assert_same(f, s)


def test_v152k_full_size_fused_equals_two_calls():
    """K = 6 (25 groups of 6 CTAs), V = 151936, low-overlap rows, WTV at T = 1.5."""
    t, d, _ = synth.make_logits("v152k", seed=0, device=DEV)
    f = FusedRun(t, d, None, S, 1.5, 0.0, 1.0)
    s = LossRun(t, d, None, S, 1.5, 0.0, 1.0)
    assert_same(f, s)
