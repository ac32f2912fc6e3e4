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

MODES = {"greedy": aal.AAL_GREEDY, "sampling": aal.AAL_SAMPLING, "both": aal.AAL_BOTH}
ORACLE_MODES = {aal.AAL_GREEDY: oracle.MODE_GREEDY, aal.AAL_SAMPLING: oracle.MODE_SAMPLING,
                aal.AAL_BOTH: oracle.MODE_BOTH}


class LossRun:
    """Forward + backward of one problem through the C ABI; results stay on the device."""

    def __init__(self, target, draft, mask, mode, T=1.0, wg=1.0, ws=1.0, dloss=1.0):
        self.prob = aal.loss_problem(draft, mode, T, wg, ws)
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


def grad_tolerance(target, draft, mask, omode, T, wg, ws, dloss, gref, nvalid, fw):
    """Per-element tolerance, widened at WTV near-ties (see module docstring)."""
    tol = GRAD_ATOL + GRAD_RTOL * np.abs(gref)
    if not (omode & oracle.MODE_SAMPLING) or nvalid == 0:
        return tol
    zp = oracle.as_f64(target)
    zq = oracle.as_f64(draft)
    lp = oracle.log_softmax(zp, T)
    lq = oracle.log_softmax(zq, T)
    amb = np.abs(lq - lp) < TIE_BAND
    amb &= (lq != lp)  # exact ties are decided identically on both sides
    if not amb.any():
        return tol
    qt = np.exp(lq)
    dEs = oracle.expected_length_partials(fw["a_s"], fw["kn"])
    B = np.abs(dloss * ws * dEs / nvalid / T)[..., None]
    dq = np.sum(np.where(amb, qt, 0.0), axis=-1, keepdims=True)
    return tol + B * qt * (amb + dq)


def check_loss(run: LossRun, target, draft, mask, mode, T, wg, ws, dloss=1.0, windows=None,
               n_windows_total=None):
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
    fw = oracle.loss_forward(t_h, d_h, m_h, omode, T, wg, ws, n_windows_total)
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
    gref = oracle.loss_backward(t_h, d_h, m_h, omode, T, wg, ws, dloss, n_windows_total)
    g = run.grad.cpu().double().numpy()[sel]
    tol = grad_tolerance(t_h, d_h, m_h, omode, T, wg, ws, dloss, gref, nvalid, fw)
    bad = np.abs(g - gref) > tol
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
