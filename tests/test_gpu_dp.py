"""Data-parallel normalisers (aal_problem / aal_seq_problem global_counts, through the C ABI).

A batch split over "ranks" (here: consecutive calls on slices of one batch), each call given |W|
and |P| of the whole batch, must reproduce the whole batch's gradient rows and per-window
expected lengths bit for bit (every per-row quantity is row-local and the scales are the same
floats), and the ranks' losses must sum to the whole batch's loss (Sec. 3.2: one 1/|W| over the
whole batch).  Checked for the two calls, the fused call and the sequence layout, with masks,
uneven shards and a shard with no valid window.
"""

import pytest
import torch

import paper_2609_24150_gb300 as aal
import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(autouse=True, scope="module")
def _fuse_short_rows():
    """The fused kernels on every row they take, short rows included (the default sends rows
    shorter than 128 KB to the two calls, which are faster there); restored afterwards."""
    aal.aal_debug_fused_min_row_bytes(0)
    yield
    aal.aal_debug_fused_min_row_bytes(-1)


G, S, B, KL = aal.AAL_GREEDY, aal.AAL_SAMPLING, aal.AAL_BOTH, aal.AAL_KL


def _bits(x):
    return x.view(torch.int16) if x.element_size() == 2 else x.view(torch.int32)


def _run(prob, draft, target, mask, fused, dloss):
    ws = torch.empty(aal.aal_workspace_size(prob), dtype=torch.uint8, device=DEV)
    N = draft.shape[0]
    loss = torch.full((1,), float("nan"), device=DEV)
    eal = torch.full((max(N, 1), 2), float("nan"), device=DEV)
    grad = torch.full_like(draft, float("nan"))
    if fused:
        aal.aal_loss_fwd_bwd(prob, draft, target, mask, ws, dloss, loss, grad, eal if N else None)
    else:
        aal.aal_loss_fwd(prob, draft, target, mask, ws, loss, eal if N else None)
        aal.aal_loss_bwd(prob, draft, target, mask, ws, dloss, grad)
    torch.cuda.synchronize()
    assert aal.aal_check_device_status(ws) == aal.AAL_OK
    return loss.item(), eal[:N], grad


@pytest.mark.parametrize("mode,T,wg,ws", [(B, 1.0, 0.5, 0.5), (KL | G, 1.0, 0.1, 0.0), (S, 1.5, 0.0, 1.0),
                                         (KL | B, 0.8, 0.3, 0.6)])
@pytest.mark.parametrize("fused", [False, True])
@pytest.mark.parametrize("dtype,V", [(torch.bfloat16, 4104), (torch.float32, 1000)])
def test_windows_sharded_over_ranks(mode, T, wg, ws, fused, dtype, V):
    N, K = 40, 5
    t, d, _ = synth.make_logits("tiny", seed=3, N=N, K=K, V=V, dtype=dtype)
    g = torch.Generator().manual_seed(4)
    mask = (torch.rand((N, K), generator=g) >= 0.15).to(torch.uint8)
    mask[0, 0] = 0
    mask[20:26, 0] = 0                         # the third shard below has no valid window
    t, d, mask = t.to(DEV), d.to(DEV), mask.to(DEV)
    nW = int((mask[:, 0] != 0).sum().item())
    nP = int((mask != 0).sum().item())
    dloss = float(nW)
    whole = _run(aal.loss_problem(d, mode, T, wg, ws, 1.0), d, t, mask, fused, dloss)
    losses, eals, grads = [], [], []
    for lo, hi in ((0, 17), (17, 20), (20, 26), (26, N)):
        p = aal.loss_problem(d[lo:hi], mode, T, wg, ws, 1.0, n_windows_global=nW, n_positions_global=nP)
        l, e, gr = _run(p, d[lo:hi].contiguous(), t[lo:hi].contiguous(), mask[lo:hi].contiguous(), fused, dloss)
        losses.append(l)
        eals.append(e)
        grads.append(gr)
    assert losses[2] == 0.0 or (mode & KL)     # no valid window: only the anchor term can remain
    assert torch.equal(_bits(torch.cat(grads)), _bits(whole[2]))
    assert torch.equal(_bits(torch.cat(eals)), _bits(whole[1]))
    assert abs(sum(losses) - whole[0]) <= 1e-6 * abs(whole[0]) + 1e-7, (sum(losses), whole[0])


def _seq_fwd_bwd(p, d, t, m, w, loss, grad, dloss, fused):
    if fused:
        aal.aal_seq_loss_fwd_bwd(p, d, t, m, w, dloss, loss, grad)
    else:
        aal.aal_seq_loss_fwd(p, d, t, m, w, loss)
        aal.aal_seq_loss_bwd(p, d, t, m, w, dloss, grad)


@pytest.mark.parametrize("fused", [False, True])
def test_sequences_sharded_over_ranks(fused):
    """The sequence layout sharded by whole sequences (L_KL + 0.1 L_EAL and EAL + WTV), as two calls
    (fp32 rows) and as the one-call form (bf16 rows, the fused kernel)."""
    if fused:
        target, draft, mask = synth.make_seq_logits("seq_tiny", seed=13, V=4104, dtype=torch.bfloat16)
    else:
        target, draft, mask = synth.make_seq_logits("seq_tiny", seed=13)
    t, d, m = target.to(DEV), draft.to(DEV), mask.to(DEV)
    Bn, Tn, V = d.shape
    K = 4
    for mode, T, wg, ws in ((KL | G, 1.0, 0.1, 0.0), (B, 1.0, 0.5, 0.5)):
        prob = aal.seq_problem(d, K, mode, T, wg, ws, False, 1.0)
        wsb = torch.empty(aal.aal_seq_workspace_size(prob), dtype=torch.uint8, device=DEV)
        loss = torch.empty(1, device=DEV)
        grad = torch.empty_like(d)
        _seq_fwd_bwd(prob, d, t, m, wsb, loss, grad, 3.0, fused)
        torch.cuda.synchronize()
        nW = nP = int((m != 0).sum().item())       # every valid position starts a window in W
        parts, total = [], 0.0
        for lo, hi in ((0, 1), (1, Bn)):
            p = aal.seq_problem(d[lo:hi], K, mode, T, wg, ws, False, 1.0, n_windows_global=nW,
                                n_positions_global=nP)
            w2 = torch.empty(aal.aal_seq_workspace_size(p), dtype=torch.uint8, device=DEV)
            l2 = torch.empty(1, device=DEV)
            g2 = torch.empty_like(d[lo:hi])
            _seq_fwd_bwd(p, d[lo:hi].contiguous(), t[lo:hi].contiguous(), m[lo:hi].contiguous(), w2, l2, g2, 3.0,
                         fused)
            torch.cuda.synchronize()
            assert aal.aal_check_device_status(w2) == aal.AAL_OK
            parts.append(g2)
            total += l2.item()
        assert torch.equal(_bits(torch.cat(parts)), _bits(grad))
        assert abs(total - loss.item()) <= 1e-6 * abs(loss.item()) + 1e-7, (total, loss.item())
