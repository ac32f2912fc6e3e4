"""Helpers for GPU-vs-oracle parity: run the C ABI on device tensors, compare with the oracle.

Tolerances (stated once, used by every GPU test):
  losses and per-window expected lengths: |got - ref| <= 1e-4 |ref| + 1e-6;
  gradients, per element: |g - g_ref| <= 1e-5 + 1e-2 |g_ref|  (bf16 output rounding is
  2^-9 relative, fp32 accumulation adds ~1e-6), widened only at near-ties of the WTV
  subgradient: where |log q~_u - log p~_u| < 1e-5 in fp64 the kernel's fp32 comparison
  may pick either side, so element u may move by g^s/T q~_u and every element of the
  row by g^s/T q~_v times the ambiguous mass;
  argmax, x*, tau: bit-exact.
"""

from __future__ import annotations

import numpy as np
import torch

import oracle
import paper_2609_24150_gb300 as aal

LOSS_RTOL = 1e-4
LOSS_ATOL = 1e-6
GRAD_ATOL = 1e-5
GRAD_RTOL = 1e-2
TIE_BAND = 1e-5

# What the widened bands set aside, per test (reset by the autouse fixture in conftest.py):
#   elems / tie_elems: gradient elements compared, and those whose fp64 log-probabilities lie
#     within TIE_BAND of each other without being equal (their subgradient side is ambiguous);
#   rescued: elements outside the unwidened tolerance that the widening accepted;
#   windows / thr_windows: reward windows compared, and those set aside because a draw that
#     decided their leading run lies within the threshold band of the reward tests.
BAND = {"elems": 0, "tie_elems": 0, "rescued": 0, "windows": 0, "thr_windows": 0}
BAND_LIMITS = {"tie": 1e-3, "rescued": 1e-3, "thr": 1e-2}


def band_reset():
    for k in BAND:
        BAND[k] = 0


def note_thr(set_aside, total):
    BAND["thr_windows"] += int(set_aside)
    BAND["windows"] += int(total)


def band_shares():
    e, w = max(BAND["elems"], 1), max(BAND["windows"], 1)
    return {"tie": BAND["tie_elems"] / e, "rescued": BAND["rescued"] / e, "thr": BAND["thr_windows"] / w}


def assert_bands():
    """The widened bands set aside at most BAND_LIMITS of what a test compared: a systematic
    error near the ties or thresholds would show up as far more."""
    sh = band_shares()
    for k, lim in BAND_LIMITS.items():
        assert sh[k] <= lim, f"band {k}: {sh[k]:.3g} of the compared items (limit {lim}); counts {BAND}"


MODES = {"greedy": aal.AAL_GREEDY, "sampling": aal.AAL_SAMPLING, "both": aal.AAL_BOTH}
# the C modes are bit sets with the oracle's values: 1 EAL, 2 WTV, 4 the KL anchor, 16 the TV term
ORACLE_MODES = {m: (oracle.MODE_GREEDY if m & aal.AAL_GREEDY else 0)
                | (oracle.MODE_SAMPLING if m & aal.AAL_SAMPLING else 0)
                | (oracle.MODE_KL if m & aal.AAL_KL else 0)
                | (oracle.MODE_TV if m & aal.AAL_TV else 0) for m in range(1, 32) if m & ~aal.AAL_GRPO}


class LossRun:
    """Forward + backward of one problem through the C ABI; results stay on the device."""

    def __init__(self, target, draft, mask, mode, T=1.0, wg=1.0, ws=1.0, dloss=1.0, wkl=1.0, wtv=1.0):
        self.prob = aal.loss_problem(draft, mode, T, wg, ws, wkl, wtv)
        self.ws_buf = torch.empty(aal.aal_workspace_size(self.prob), dtype=torch.uint8,
                                  device=draft.device)
        N = draft.shape[0]
        self.loss = torch.full((1,), float("nan"), dtype=torch.float32, device=draft.device)
        self.eal = torch.full((max(N, 1), 2), float("nan"), dtype=torch.float32, device=draft.device)
        self.grad = torch.full_like(draft, float("nan"))
        aal.aal_loss_fwd(self.prob, draft, target, mask, self.ws_buf, self.loss,
                         self.eal if N > 0 else None)
        aal.aal_loss_bwd(self.prob, draft, target, mask, self.ws_buf, dloss, self.grad)
        torch.cuda.synchronize()
        assert aal.aal_check_device_status(self.ws_buf) == aal.AAL_OK


def grad_tolerance(target, draft, mask, omode, T, wg, ws, dloss, gref, nvalid, fw, wtv=0.0):
    """Per-element tolerance, widened at WTV / TV near-ties (see module docstring)."""
    tol = GRAD_ATOL + GRAD_RTOL * np.abs(gref)
    BAND["elems"] += int(np.prod(np.shape(gref)))
    if not (omode & (oracle.MODE_SAMPLING | oracle.MODE_TV)) or nvalid == 0:
        return tol
    zp = oracle.as_f64(target)
    zq = oracle.as_f64(draft)
    lp = oracle.log_softmax(zp, T)
    lq = oracle.log_softmax(zq, T)
    amb = np.abs(lq - lp) < TIE_BAND
    amb &= (lq != lp)  # exact ties are decided identically on both sides
    BAND["tie_elems"] += int(amb.sum())
    if not amb.any():
        return tol
    qt = np.exp(lq)
    kn = fw["kn"]
    coef = np.zeros(amb.shape[:-1])
    if omode & oracle.MODE_SAMPLING:
        coef = coef + ws * oracle.expected_length_partials(fw["a_s"], kn)
    if omode & oracle.MODE_TV:
        depth = np.arange(coef.shape[-1])[None, :]
        coef = coef + np.where(depth < kn[:, None], wtv / np.maximum(kn, 1)[:, None], 0.0)
    B = np.abs(dloss * coef / nvalid / T)[..., None]
    dq = np.sum(np.where(amb, qt, 0.0), axis=-1, keepdims=True)
    return tol + B * qt * (amb + dq)


def check_loss(run: LossRun, target, draft, mask, mode, T, wg, ws, dloss=1.0, windows=None,
               n_windows_total=None, wkl=1.0, n_positions_total=None, wtv=1.0):
    """Compare loss / eal / gradient of ``run`` with the oracle (optionally on some windows)."""
    omode = ORACLE_MODES[mode]
    if windows is None:
        t_h, d_h = target.cpu(), draft.cpu()
        m_h = None if mask is None else mask.cpu().numpy()
        sel = slice(None)
    else:
        idx = torch.as_tensor(windows, device=target.device)
        t_h, d_h = target[idx].cpu(), draft[idx].cpu()
        m_h = None if mask is None else mask[idx].cpu().numpy()
        sel = np.asarray(windows)
    fw = oracle.objective_forward(t_h, d_h, m_h, omode, T, wg, ws, wkl, n_windows_total, n_positions_total, wtv)
    nvalid = fw["nvalid"]
    eal = run.eal.cpu().numpy()[sel]
    if omode & oracle.MODE_GREEDY:
        np.testing.assert_allclose(eal[:, 0], fw["eal_g"], rtol=LOSS_RTOL, atol=LOSS_ATOL)
    if omode & oracle.MODE_SAMPLING:
        np.testing.assert_allclose(eal[:, 1], fw["eal_s"], rtol=LOSS_RTOL, atol=LOSS_ATOL)
    if windows is None:
        ref = fw["loss"]
        got = float(run.loss.item())
        assert abs(got - ref) <= LOSS_RTOL * abs(ref) + LOSS_ATOL, (got, ref)
    gref = oracle.objective_backward(t_h, d_h, m_h, omode, T, wg, ws, wkl, dloss, n_windows_total,
                                     n_positions_total, wtv)
    g = run.grad.cpu().double().numpy()[sel]
    tol = grad_tolerance(t_h, d_h, m_h, omode, T, wg, ws, dloss, gref, nvalid, fw, wtv if omode & oracle.MODE_TV else 0.0)
    bad = np.abs(g - gref) > tol
    BAND["rescued"] += int(np.sum((np.abs(g - gref) > GRAD_ATOL + GRAD_RTOL * np.abs(gref)) & ~bad))
    if bad.any():
        i = tuple(np.argwhere(bad)[0])
        raise AssertionError(f"{int(bad.sum())} gradient elements off; first {i}: "
                             f"gpu {g[i]!r} oracle {gref[i]!r} tol {tol[i]!r}")
    return fw


def loss_from_eal(run: LossRun, mode, wg, ws, nvalid):
    """The loss the per-window outputs imply: -(w_g sum E^g + w_s sum E^s) / |W|."""
    eal = run.eal.double().cpu().numpy()
    num = 0.0
    if mode & aal.AAL_GREEDY:
        num += wg * eal[:, 0].sum()
    if mode & aal.AAL_SAMPLING:
        num += ws * eal[:, 1].sum()
    return -num / nvalid if nvalid else 0.0


# -------------------------------------------------------------------------- sequence layout

class SeqRun:
    """Forward + backward of one sequence-layout problem through the C ABI (two calls, or the
    one-call aal_seq_loss_fwd_bwd with ``fused``)."""

    def __init__(self, target, draft, mask, K, mode, T=1.0, wg=1.0, ws=1.0, dloss=1.0, full_windows=False,
                 wkl=1.0, wtv=1.0, fused=False):
        self.prob = aal.seq_problem(draft, K, mode, T, wg, ws, full_windows, wkl, wtv)
        self.ws_buf = torch.empty(aal.aal_seq_workspace_size(self.prob), dtype=torch.uint8,
                                  device=draft.device)
        R = draft.shape[0] * draft.shape[1]
        self.loss = torch.full((1,), float("nan"), dtype=torch.float32, device=draft.device)
        self.eal = torch.full((max(R, 1), 2), float("nan"), dtype=torch.float32, device=draft.device)
        self.grad = torch.full_like(draft, float("nan"))
        if fused:   # aal_seq_loss_fwd_bwd: one call
            aal.aal_seq_loss_fwd_bwd(self.prob, draft, target, mask, self.ws_buf, dloss, self.loss, self.grad,
                                     self.eal if R > 0 else None)
        else:
            aal.aal_seq_loss_fwd(self.prob, draft, target, mask, self.ws_buf, self.loss,
                                 self.eal if R > 0 else None)
            aal.aal_seq_loss_bwd(self.prob, draft, target, mask, self.ws_buf, dloss, self.grad)
        torch.cuda.synchronize()
        assert aal.aal_check_device_status(self.ws_buf) == aal.AAL_OK


def seq_grad_tolerance(target, draft, mask, K, omode, T, wg, ws, dloss, gref, nvalid_total,
                       full_windows=False, wtv=0.0):
    """Per-position tolerance: GRAD_ATOL + GRAD_RTOL |g_ref| plus the near-tie widening of every
    window row the position contributes to."""
    wp, wq, wm, src = oracle.gather_windows(target, draft, mask, K, full_windows)
    fw = oracle.loss_forward(wp, wq, wm, omode, T, wg, ws, nvalid_total)
    widen = grad_tolerance(wp, wq, wm, omode, T, wg, ws, dloss, np.zeros(wq.shape), nvalid_total,
                           fw, wtv) - GRAD_ATOL
    Bq, Tq, V = gref.shape
    extra = np.zeros((Bq * Tq, V))
    for n, j in np.argwhere(src >= 0):
        extra[src[n, j]] += widen[n, j]
    return GRAD_ATOL + GRAD_RTOL * np.abs(gref) + extra.reshape(Bq, Tq, V)


def _assert_grad(g, gref, tol, where=""):
    bad = np.abs(g - gref) > tol
    BAND["rescued"] += int(np.sum((np.abs(g - gref) > GRAD_ATOL + GRAD_RTOL * np.abs(gref)) & ~bad))
    if bad.any():
        i = tuple(np.argwhere(bad)[0])
        raise AssertionError(f"{where}{int(bad.sum())} gradient elements off; first {i}: "
                             f"gpu {g[i]!r} oracle {gref[i]!r} tol {tol[i]!r}")


def check_seq_loss(run: SeqRun, target, draft, mask, K, mode, T, wg, ws, dloss=1.0, full_windows=False,
                   wkl=1.0, wtv=1.0):
    """Every output of a sequence-layout run against the oracle on all positions."""
    omode = ORACLE_MODES[mode]
    t_h, d_h = target.cpu(), draft.cpu()
    m_h = None if mask is None else mask.cpu().numpy()
    fw = oracle.seq_objective_forward(t_h, d_h, m_h, K, omode, T, wg, ws, wkl, full_windows=full_windows,
                                      w_tv=wtv)
    eal = run.eal.cpu().numpy()
    if omode & oracle.MODE_GREEDY:
        np.testing.assert_allclose(eal[:, 0], fw["eal_g"], rtol=LOSS_RTOL, atol=LOSS_ATOL)
    if omode & oracle.MODE_SAMPLING:
        np.testing.assert_allclose(eal[:, 1], fw["eal_s"], rtol=LOSS_RTOL, atol=LOSS_ATOL)
    got, ref = float(run.loss.item()), fw["loss"]
    assert abs(got - ref) <= LOSS_RTOL * abs(ref) + LOSS_ATOL, (got, ref)
    gref = oracle.seq_objective_backward(t_h, d_h, m_h, K, omode, T, wg, ws, wkl, dloss,
                                         full_windows=full_windows, w_tv=wtv)
    tol = seq_grad_tolerance(t_h, d_h, m_h, K, omode, T, wg, ws, dloss, gref, fw["nvalid"], full_windows,
                             wtv if omode & oracle.MODE_TV else 0.0)
    _assert_grad(run.grad.cpu().double().numpy(), gref, tol)
    return fw


def check_seq_positions(run: SeqRun, target, draft, mask, K, mode, T, wg, ws, dloss, positions,
                        nvalid_total, wkl=1.0, npos_total=None):
    """Sampled check at full size: for each (b, t) the oracle runs on positions t-K+1 .. t+K-1 of
    sequence b only (every window containing t, and the window starting at t, lie inside), with
    |W| (and the anchor's |positions|) of the whole batch; the window starting at t and the
    gradient row of t are compared."""
    omode = ORACLE_MODES[mode]
    Tn = draft.shape[1]
    eal = run.eal.view(draft.shape[0], Tn, 2)
    for b, t in positions:
        lo, hi = max(0, t - K + 1), min(Tn, t + K)
        t_h = target[b:b + 1, lo:hi].cpu()
        d_h = draft[b:b + 1, lo:hi].cpu()
        m_h = None if mask is None else mask[b:b + 1, lo:hi].cpu().numpy()
        fw = oracle.seq_objective_forward(t_h, d_h, m_h, K, omode, T, wg, ws, wkl, nvalid_total, npos_total)
        e = eal[b, t].cpu().numpy()
        if omode & oracle.MODE_GREEDY:
            np.testing.assert_allclose(e[0], fw["eal_g"][t - lo], rtol=LOSS_RTOL, atol=LOSS_ATOL)
        if omode & oracle.MODE_SAMPLING:
            np.testing.assert_allclose(e[1], fw["eal_s"][t - lo], rtol=LOSS_RTOL, atol=LOSS_ATOL)
        gref = oracle.seq_objective_backward(t_h, d_h, m_h, K, omode, T, wg, ws, wkl, dloss, nvalid_total,
                                             npos_total)
        tol = seq_grad_tolerance(t_h, d_h, m_h, K, omode, T, wg, ws, dloss, gref, nvalid_total)
        g = run.grad[b, t].cpu().double().numpy()
        _assert_grad(g, gref[0, t - lo], tol[0, t - lo], where=f"position ({b}, {t}): ")


def seq_window_counts(mask, B, Tn):
    """|W| of a sequence batch: the number of valid positions (each starts one window)."""
    return B * Tn if mask is None else int(mask.sum().item())
