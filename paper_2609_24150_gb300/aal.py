"""ctypes binding of libaal.so: same names as the C ABI, argument marshalling only."""

from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

AAL_OK = 0
AAL_ERR_INVALID_ARG = 1
AAL_ERR_UNSUPPORTED = 2
AAL_ERR_WORKSPACE = 3
AAL_ERR_CUDA = 4
AAL_ERR_TIMEOUT = 5

AAL_F32 = 0
AAL_BF16 = 1

AAL_GREEDY = 1
AAL_SAMPLING = 2
AAL_BOTH = 3
AAL_KL = 4          # mode bit: the forward-KL anchor
AAL_GRPO = 8        # mode bit: the backward adds the GRPO surrogate's gradient
AAL_TV = 16         # mode bit: the L_TV baseline's window-averaged TV term
AAL_IDS = 32        # mode bit: `target` holds int32 token ids (x*), not logits
AAL_SAMPLED_DRAFT = 4   # reward mode flag (with AAL_SAMPLING): the drafted token is drawn from q~

AAL_MAX_K = 8
AAL_NOALLOC_MAX_ROWS = 1 << 20   # N * K limit of aal_accept_reward_noalloc

_HERE = os.path.dirname(os.path.abspath(__file__))


def library_path() -> str:
    return os.path.join(_HERE, "libaal.so")


class AalProblem(ctypes.Structure):
    """Mirror of ``aal_problem``."""
    _fields_ = [("N", ctypes.c_int64), ("K", ctypes.c_int64), ("V", ctypes.c_int64),
                ("dtype", ctypes.c_int32), ("mode", ctypes.c_int32),
                ("temperature", ctypes.c_float), ("w_greedy", ctypes.c_float),
                ("w_sampling", ctypes.c_float), ("w_kl", ctypes.c_float), ("w_tv", ctypes.c_float),
                ("global_counts", ctypes.c_int32), ("n_windows_global", ctypes.c_int64),
                ("n_positions_global", ctypes.c_int64)]


class AalRewardProblem(ctypes.Structure):
    """Mirror of ``aal_reward_problem``."""
    _fields_ = [("N", ctypes.c_int64), ("K", ctypes.c_int64), ("V", ctypes.c_int64),
                ("dtype", ctypes.c_int32), ("mode", ctypes.c_int32),
                ("temperature", ctypes.c_float), ("adv_clip", ctypes.c_float),
                ("seed", ctypes.c_uint64), ("row_offset", ctypes.c_int64),
                ("windows_per_rollout", ctypes.c_int64), ("rollouts_per_group", ctypes.c_int64)]


class AalSeqProblem(ctypes.Structure):
    """Mirror of ``aal_seq_problem``."""
    _fields_ = [("B", ctypes.c_int64), ("seq_len", ctypes.c_int64), ("K", ctypes.c_int64),
                ("V", ctypes.c_int64), ("dtype", ctypes.c_int32), ("mode", ctypes.c_int32),
                ("temperature", ctypes.c_float), ("w_greedy", ctypes.c_float),
                ("w_sampling", ctypes.c_float), ("w_kl", ctypes.c_float), ("w_tv", ctypes.c_float),
                ("full_windows", ctypes.c_int32), ("global_counts", ctypes.c_int32),
                ("n_windows_global", ctypes.c_int64), ("n_positions_global", ctypes.c_int64)]


class AalGrpoProblem(ctypes.Structure):
    """Mirror of ``aal_grpo_problem``."""
    _fields_ = [("N", ctypes.c_int64), ("K", ctypes.c_int64), ("V", ctypes.c_int64),
                ("dtype", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("windows_per_rollout", ctypes.c_int64), ("rollouts_per_group", ctypes.c_int64),
                ("adv_clip", ctypes.c_float), ("eps_clip", ctypes.c_float),
                ("rho_min", ctypes.c_float), ("rho_max", ctypes.c_float),
                ("log_rho_clip", ctypes.c_float), ("w_grpo", ctypes.c_float)]


class AalError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {aal_status_string(code)}")


_LIB = None


def library() -> ctypes.CDLL:
    """Load libaal.so once; raise ImportError if it has not been built."""
    global _LIB
    if _LIB is not None:
        return _LIB
    path = library_path()
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with `python -m paper_2609_24150_gb300.build`")
    lib = ctypes.CDLL(path)
    vp, sz = ctypes.c_void_p, ctypes.c_size_t
    P = ctypes.POINTER(AalProblem)
    RP = ctypes.POINTER(AalRewardProblem)
    lib.aal_workspace_size.argtypes = [P, ctypes.POINTER(sz)]
    lib.aal_reward_workspace_size.argtypes = [RP, ctypes.POINTER(sz)]
    lib.aal_loss_fwd.argtypes = [P, vp, vp, vp, vp, sz, vp, vp, vp]
    lib.aal_loss_bwd.argtypes = [P, vp, vp, vp, vp, sz, ctypes.c_float, vp, vp]
    lib.aal_loss_fwd_bwd.argtypes = [P, vp, vp, vp, vp, sz, ctypes.c_float, vp, vp, vp, vp]
    lib.aal_accept_reward.argtypes = [RP, vp, vp, vp, vp, sz, vp, vp, vp, vp, vp]
    lib.aal_accept_reward_noalloc.argtypes = [RP, vp, vp, vp, vp, vp, vp, vp, vp]
    lib.aal_accept_reward_from_loss.argtypes = [RP, P, vp, sz, vp, sz, vp, vp, vp, vp]
    lib.aal_accept_reward_sampled_from_loss.argtypes = [RP, P, vp, vp, vp, sz, vp, sz, vp, vp, vp, vp]
    SP = ctypes.POINTER(AalSeqProblem)
    lib.aal_seq_workspace_size.argtypes = [SP, ctypes.POINTER(sz)]
    lib.aal_seq_loss_fwd.argtypes = [SP, vp, vp, vp, vp, sz, vp, vp, vp]
    lib.aal_seq_loss_bwd.argtypes = [SP, vp, vp, vp, vp, sz, ctypes.c_float, vp, vp]
    lib.aal_seq_loss_fwd_bwd.argtypes = [SP, vp, vp, vp, vp, sz, ctypes.c_float, vp, vp, vp, vp]
    GP = ctypes.POINTER(AalGrpoProblem)
    lib.aal_grpo_workspace_size.argtypes = [GP, ctypes.POINTER(sz)]
    lib.aal_grpo_from_loss.argtypes = [GP, P, vp, sz, vp, vp, sz, vp, vp, vp, vp, vp, vp]
    lib.aal_seq_grpo_workspace_size.argtypes = [GP, SP, ctypes.POINTER(sz)]
    lib.aal_seq_grpo_from_loss.argtypes = [GP, SP, vp, sz, vp, vp, vp, sz, vp, vp, vp, vp, vp, vp]
    lib.aal_check_device_status.argtypes = [vp, vp]
    lib.aal_debug_fail_next_forward.argtypes = [ctypes.c_int64, ctypes.c_uint64]
    lib.aal_debug_fail_next_forward.restype = None
    lib.aal_debug_solo_windows.argtypes = [ctypes.c_int64, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32]
    lib.aal_debug_solo_windows.restype = ctypes.c_int64
    lib.aal_debug_fused_min_row_bytes.argtypes = [ctypes.c_int64]
    lib.aal_debug_fused_min_row_bytes.restype = None
    lib.aal_status_string.argtypes = [ctypes.c_int]
    lib.aal_status_string.restype = ctypes.c_char_p
    lib.aal_abi_version.argtypes = []
    lib.aal_abi_version.restype = ctypes.c_int32
    for f in ("aal_workspace_size", "aal_reward_workspace_size", "aal_loss_fwd", "aal_loss_bwd", "aal_loss_fwd_bwd",
              "aal_accept_reward", "aal_accept_reward_noalloc", "aal_accept_reward_from_loss",
              "aal_accept_reward_sampled_from_loss", "aal_seq_workspace_size", "aal_seq_loss_fwd",
              "aal_seq_loss_bwd", "aal_seq_loss_fwd_bwd", "aal_check_device_status",
              "aal_grpo_workspace_size", "aal_grpo_from_loss", "aal_seq_grpo_workspace_size",
              "aal_seq_grpo_from_loss"):
        getattr(lib, f).restype = ctypes.c_int
    _LIB = lib
    return lib


# -------------------------------------------------------------------------- marshalling

_DTYPES = {torch.float32: AAL_F32, torch.bfloat16: AAL_BF16}


def _ptr(x, what: str, dtype=None, numel=None) -> Optional[int]:
    """Device address of a CUDA tensor (or a raw int address); None stays NULL."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if not isinstance(x, torch.Tensor):
        raise TypeError(f"{what}: expected a CUDA tensor or an address, got {type(x)}")
    if not x.is_cuda:
        raise ValueError(f"{what}: tensor must be on a CUDA device (libaal has no CPU path)")
    if not x.is_contiguous():
        raise ValueError(f"{what}: tensor must be contiguous")
    if dtype is not None and x.dtype != dtype:
        raise ValueError(f"{what}: expected {dtype}, got {x.dtype}")
    if numel is not None and x.numel() < numel:
        raise ValueError(f"{what}: needs at least {numel} elements, has {x.numel()}")
    return x.data_ptr()


def _nbytes(x) -> int:
    return x.numel() * x.element_size() if isinstance(x, torch.Tensor) else 0


def _stream(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _check(code: int, where: str):
    if code != AAL_OK:
        raise AalError(code, where)


def _global(n_windows_global, n_positions_global):
    """(global_counts, |W|, |P|) fields: both counts given, or neither (this call's own)."""
    if (n_windows_global is None) != (n_positions_global is None):
        raise ValueError("give both global counts (|W| and |P| of the whole batch) or neither")
    if n_windows_global is None:
        return 0, 0, 0
    return 1, int(n_windows_global), int(n_positions_global)


def loss_problem(draft: torch.Tensor, mode: int, temperature: float = 1.0, w_greedy: float = 1.0,
                 w_sampling: float = 1.0, w_kl: float = 1.0, w_tv: float = 1.0,
                 n_windows_global: Optional[int] = None, n_positions_global: Optional[int] = None) -> AalProblem:
    """Problem struct for [N][K][V] logits (``w_kl`` weighs the AAL_KL anchor, ``w_tv`` the
    AAL_TV term).  ``n_windows_global`` / ``n_positions_global``: |W| and |P| of a whole
    data-parallel batch that this call is one shard of (the loss and gradient are normalised by
    them instead of the shard's own)."""
    if draft.dim() != 3:
        raise ValueError("logits must be [N][K][V]")
    N, K, V = draft.shape
    if draft.dtype not in _DTYPES:
        raise ValueError(f"unsupported dtype {draft.dtype}")
    return AalProblem(N, K, V, _DTYPES[draft.dtype], mode, temperature, w_greedy, w_sampling, w_kl, w_tv,
                      *_global(n_windows_global, n_positions_global))


def seq_problem(draft: torch.Tensor, K: int, mode: int, temperature: float = 1.0, w_greedy: float = 1.0,
                w_sampling: float = 1.0, full_windows: bool = False, w_kl: float = 1.0,
                w_tv: float = 1.0, n_windows_global: Optional[int] = None,
                n_positions_global: Optional[int] = None) -> AalSeqProblem:
    """Problem struct for [B][seq_len][V] logits with sliding windows of K positions
    (``full_windows``: only windows with all K positions valid belong to W; the global counts
    as in loss_problem, for a batch sharded by whole sequences)."""
    if draft.dim() != 3:
        raise ValueError("logits must be [B][seq_len][V]")
    B, S, V = draft.shape
    if draft.dtype not in _DTYPES:
        raise ValueError(f"unsupported dtype {draft.dtype}")
    return AalSeqProblem(B, S, K, V, _DTYPES[draft.dtype], mode, temperature, w_greedy, w_sampling,
                         w_kl, w_tv, int(bool(full_windows)), *_global(n_windows_global, n_positions_global))


def reward_problem(draft: torch.Tensor, mode: int, temperature: float = 1.0, adv_clip: float = 5.0,
                   seed: int = 0, row_offset: int = 0, windows_per_rollout: int = 1,
                   rollouts_per_group: int = 1) -> AalRewardProblem:
    if draft.dim() != 3:
        raise ValueError("logits must be [N][K][V]")
    N, K, V = draft.shape
    return AalRewardProblem(N, K, V, _DTYPES[draft.dtype], mode, temperature, adv_clip, seed,
                            row_offset, windows_per_rollout, rollouts_per_group)


# -------------------------------------------------------------------------- the C ABI

def aal_status_string(code: int) -> str:
    return library().aal_status_string(int(code)).decode()


def aal_abi_version() -> int:
    return int(library().aal_abi_version())


def aal_workspace_size(problem: AalProblem) -> int:
    out = ctypes.c_size_t(0)
    _check(library().aal_workspace_size(ctypes.byref(problem), ctypes.byref(out)), "aal_workspace_size")
    return out.value


def aal_reward_workspace_size(problem: AalRewardProblem) -> int:
    out = ctypes.c_size_t(0)
    _check(library().aal_reward_workspace_size(ctypes.byref(problem), ctypes.byref(out)),
           "aal_reward_workspace_size")
    return out.value


def aal_loss_fwd(problem: AalProblem, draft, target, mask, workspace, loss, eal=None, stream=None):
    """Forward of the EAL / WTV loss; writes loss[0] (and eal[N][2] when given)."""
    N = problem.N
    code = library().aal_loss_fwd(
        ctypes.byref(problem), _ptr(draft, "draft"), _ptr(target, "target"),
        _ptr(mask, "mask", torch.uint8, N * problem.K), _ptr(workspace, "workspace"),
        _nbytes(workspace), _ptr(loss, "loss", torch.float32, 1),
        _ptr(eal, "eal", torch.float32, 2 * N), _stream(stream))
    _check(code, "aal_loss_fwd")


def aal_loss_bwd(problem: AalProblem, draft, target, mask, workspace, dloss: float, grad, stream=None):
    """Backward: grad = dloss * dL/d draft, in the draft's dtype."""
    code = library().aal_loss_bwd(
        ctypes.byref(problem), _ptr(draft, "draft"), _ptr(target, "target"),
        _ptr(mask, "mask", torch.uint8), _ptr(workspace, "workspace"), _nbytes(workspace),
        float(dloss), _ptr(grad, "grad"), _stream(stream))
    _check(code, "aal_loss_bwd")


def aal_loss_fwd_bwd(problem: AalProblem, draft, target, mask, workspace, dloss: float, loss, grad, eal=None,
                     stream=None):
    """Forward and backward in one call: loss[0] (and eal[N][2]) as aal_loss_fwd, grad as
    aal_loss_bwd with the same dloss; the logits are read from HBM once."""
    N = problem.N
    code = library().aal_loss_fwd_bwd(
        ctypes.byref(problem), _ptr(draft, "draft"), _ptr(target, "target"),
        _ptr(mask, "mask", torch.uint8, N * problem.K), _ptr(workspace, "workspace"),
        _nbytes(workspace), float(dloss), _ptr(loss, "loss", torch.float32, 1),
        _ptr(eal, "eal", torch.float32, 2 * N), _ptr(grad, "grad"), _stream(stream))
    _check(code, "aal_loss_fwd_bwd")


def grpo_problem(draft: torch.Tensor, windows_per_rollout: int = 1, rollouts_per_group: int = 1,
                 adv_clip: float = 5.0, eps_clip: float = 0.2, rho_min: float = 0.0, rho_max: float = 10.0,
                 log_rho_clip: float = 10.0, w_grpo: float = 1.0) -> AalGrpoProblem:
    """GRPO problem struct for the [N][K][V] windows of a loss problem."""
    if draft.dim() != 3:
        raise ValueError("logits must be [N][K][V]")
    N, K, V = draft.shape
    return AalGrpoProblem(N, K, V, _DTYPES[draft.dtype], 0, windows_per_rollout, rollouts_per_group,
                          adv_clip, eps_clip, rho_min, rho_max, log_rho_clip, w_grpo)


def aal_grpo_workspace_size(problem: AalGrpoProblem) -> int:
    out = ctypes.c_size_t(0)
    _check(library().aal_grpo_workspace_size(ctypes.byref(problem), ctypes.byref(out)),
           "aal_grpo_workspace_size")
    return out.value


def aal_grpo_from_loss(problem: AalGrpoProblem, loss_problem_: AalProblem, loss_workspace, ref_draft,
                       workspace, grpo_loss, tau=None, tau_ref=None, advantage=None, log_rho=None,
                       stream=None):
    """GRPO stage after aal_loss_fwd (mode with AAL_GRPO): L_GRPO, tau, tau_ref, advantages,
    log rho; writes the surrogate's gradient coefficients into the loss workspace."""
    N = problem.N
    nroll = N // max(1, problem.windows_per_rollout)
    code = library().aal_grpo_from_loss(
        ctypes.byref(problem), ctypes.byref(loss_problem_), _ptr(loss_workspace, "loss_workspace"),
        _nbytes(loss_workspace), _ptr(ref_draft, "ref_draft"), _ptr(workspace, "workspace"),
        _nbytes(workspace), _ptr(grpo_loss, "grpo_loss", torch.float32, 1),
        _ptr(tau, "tau", torch.int32, N), _ptr(tau_ref, "tau_ref", torch.int32, N),
        _ptr(advantage, "advantage", torch.float32, nroll), _ptr(log_rho, "log_rho", torch.float32, N),
        _stream(stream))
    _check(code, "aal_grpo_from_loss")


def grpo_seq_problem(n_windows: int, draft: torch.Tensor, K: int, windows_per_rollout: int = 1,
                     rollouts_per_group: int = 1, adv_clip: float = 5.0, eps_clip: float = 0.2,
                     rho_min: float = 0.0, rho_max: float = 10.0, log_rho_clip: float = 10.0,
                     w_grpo: float = 1.0) -> AalGrpoProblem:
    """GRPO problem struct for n_windows windows of K positions sliced from [B][T][V] logits."""
    if draft.dim() != 3:
        raise ValueError("logits must be [B][seq_len][V]")
    V = draft.shape[2]
    return AalGrpoProblem(n_windows, K, V, _DTYPES[draft.dtype], 0, windows_per_rollout, rollouts_per_group,
                          adv_clip, eps_clip, rho_min, rho_max, log_rho_clip, w_grpo)


def aal_seq_grpo_workspace_size(problem: AalGrpoProblem, seq_problem_: AalSeqProblem) -> int:
    out = ctypes.c_size_t(0)
    _check(library().aal_seq_grpo_workspace_size(ctypes.byref(problem), ctypes.byref(seq_problem_),
                                                 ctypes.byref(out)), "aal_seq_grpo_workspace_size")
    return out.value


def aal_seq_grpo_from_loss(problem: AalGrpoProblem, seq_problem_: AalSeqProblem, loss_workspace, ref_draft,
                           starts, workspace, grpo_loss, tau=None, tau_ref=None, advantage=None, log_rho=None,
                           stream=None):
    """GRPO stage over windows sliced from sequences (ascending flat start positions), after
    aal_seq_loss_fwd with AAL_GRPO; writes the per-position gradient coefficients."""
    N = problem.N
    nroll = N // max(1, problem.windows_per_rollout)
    code = library().aal_seq_grpo_from_loss(
        ctypes.byref(problem), ctypes.byref(seq_problem_), _ptr(loss_workspace, "loss_workspace"),
        _nbytes(loss_workspace), _ptr(ref_draft, "ref_draft"), _ptr(starts, "starts", torch.int32, N),
        _ptr(workspace, "workspace"), _nbytes(workspace), _ptr(grpo_loss, "grpo_loss", torch.float32, 1),
        _ptr(tau, "tau", torch.int32, N), _ptr(tau_ref, "tau_ref", torch.int32, N),
        _ptr(advantage, "advantage", torch.float32, nroll), _ptr(log_rho, "log_rho", torch.float32, N),
        _stream(stream))
    _check(code, "aal_seq_grpo_from_loss")


def aal_seq_workspace_size(problem: AalSeqProblem) -> int:
    out = ctypes.c_size_t(0)
    _check(library().aal_seq_workspace_size(ctypes.byref(problem), ctypes.byref(out)),
           "aal_seq_workspace_size")
    return out.value


def aal_seq_loss_fwd(problem: AalSeqProblem, draft, target, mask, workspace, loss, eal=None, stream=None):
    """Forward of the loss over every sliding window of every sequence; writes loss[0] (and
    eal[B*seq_len][2] when given)."""
    R = problem.B * problem.seq_len
    code = library().aal_seq_loss_fwd(
        ctypes.byref(problem), _ptr(draft, "draft"), _ptr(target, "target"),
        _ptr(mask, "mask", torch.uint8, R), _ptr(workspace, "workspace"), _nbytes(workspace),
        _ptr(loss, "loss", torch.float32, 1), _ptr(eal, "eal", torch.float32, 2 * R), _stream(stream))
    _check(code, "aal_seq_loss_fwd")


def aal_seq_loss_bwd(problem: AalSeqProblem, draft, target, mask, workspace, dloss: float, grad, stream=None):
    """Backward of the sequence loss: grad = dloss * dL/d draft, summed over each position's windows."""
    code = library().aal_seq_loss_bwd(
        ctypes.byref(problem), _ptr(draft, "draft"), _ptr(target, "target"),
        _ptr(mask, "mask", torch.uint8), _ptr(workspace, "workspace"), _nbytes(workspace),
        float(dloss), _ptr(grad, "grad"), _stream(stream))
    _check(code, "aal_seq_loss_bwd")


def aal_seq_loss_fwd_bwd(problem: AalSeqProblem, draft, target, mask, workspace, dloss: float, loss, grad,
                         eal=None, stream=None):
    """Forward and backward of the sequence loss in one call: loss[0] (and eal[B*seq_len][2]) as
    aal_seq_loss_fwd, grad as aal_seq_loss_bwd with the same dloss; each position's logits are
    read from HBM once."""
    R = problem.B * problem.seq_len
    code = library().aal_seq_loss_fwd_bwd(
        ctypes.byref(problem), _ptr(draft, "draft"), _ptr(target, "target"),
        _ptr(mask, "mask", torch.uint8, R), _ptr(workspace, "workspace"), _nbytes(workspace),
        float(dloss), _ptr(loss, "loss", torch.float32, 1), _ptr(eal, "eal", torch.float32, 2 * R),
        _ptr(grad, "grad"), _stream(stream))
    _check(code, "aal_seq_loss_fwd_bwd")


def aal_accept_reward(problem: AalRewardProblem, draft, target, ref_draft, workspace, tau,
                      tau_ref, rollout_len, advantage, stream=None):
    """Simulated acceptance lengths, debiased rewards, rollout lengths and advantages."""
    N = problem.N
    nroll = N // max(1, problem.windows_per_rollout)
    code = library().aal_accept_reward(
        ctypes.byref(problem), _ptr(draft, "draft"), _ptr(target, "target"),
        _ptr(ref_draft, "ref_draft"), _ptr(workspace, "workspace"), _nbytes(workspace),
        _ptr(tau, "tau", torch.int32, N), _ptr(tau_ref, "tau_ref", torch.int32, N),
        _ptr(rollout_len, "rollout_len", torch.float32, nroll),
        _ptr(advantage, "advantage", torch.float32, nroll), _stream(stream))
    _check(code, "aal_accept_reward")


def aal_accept_reward_from_loss(problem: AalRewardProblem, loss_problem_: AalProblem, loss_workspace,
                                workspace, tau, rollout_len, advantage, stream=None):
    """The draft's reward from the statistics of a completed aal_loss_fwd (no logit pass)."""
    N = problem.N
    nroll = N // max(1, problem.windows_per_rollout)
    code = library().aal_accept_reward_from_loss(
        ctypes.byref(problem), ctypes.byref(loss_problem_), _ptr(loss_workspace, "loss_workspace"),
        _nbytes(loss_workspace), _ptr(workspace, "workspace"), _nbytes(workspace),
        _ptr(tau, "tau", torch.int32, N), _ptr(rollout_len, "rollout_len", torch.float32, nroll),
        _ptr(advantage, "advantage", torch.float32, nroll), _stream(stream))
    _check(code, "aal_accept_reward_from_loss")


def aal_accept_reward_sampled_from_loss(problem: AalRewardProblem, loss_problem_: AalProblem, draft, target,
                                        loss_workspace, workspace, tau, rollout_len, advantage, stream=None):
    """The sampled-draft reward with the normalisers of a completed aal_loss_fwd: the draft
    streamed once for the draws, the target read at the drawn tokens only."""
    N = problem.N
    nroll = N // max(1, problem.windows_per_rollout)
    code = library().aal_accept_reward_sampled_from_loss(
        ctypes.byref(problem), ctypes.byref(loss_problem_), _ptr(draft, "draft"), _ptr(target, "target"),
        _ptr(loss_workspace, "loss_workspace"), _nbytes(loss_workspace), _ptr(workspace, "workspace"),
        _nbytes(workspace), _ptr(tau, "tau", torch.int32, N),
        _ptr(rollout_len, "rollout_len", torch.float32, nroll),
        _ptr(advantage, "advantage", torch.float32, nroll), _stream(stream))
    _check(code, "aal_accept_reward_sampled_from_loss")


def aal_accept_reward_noalloc(problem: AalRewardProblem, draft, target, ref_draft, tau, tau_ref,
                              rollout_len, advantage, stream=None):
    """aal_accept_reward with the library's fixed scratch array instead of a workspace.

    For callers that cannot allocate device memory (e.g. their memory is fully reserved by
    their own allocator).  At most AAL_NOALLOC_MAX_ROWS = N * K rows; calls share one scratch
    array, so calls that overlap on the GPU must be ordered by the caller.
    """
    N = problem.N
    if N * problem.K > AAL_NOALLOC_MAX_ROWS:
        raise AalError(AAL_ERR_UNSUPPORTED, f"aal_accept_reward_noalloc: N*K = {N * problem.K} "
                       f"exceeds the fixed scratch limit of {AAL_NOALLOC_MAX_ROWS} rows")
    nroll = N // max(1, problem.windows_per_rollout)
    code = library().aal_accept_reward_noalloc(
        ctypes.byref(problem), _ptr(draft, "draft"), _ptr(target, "target"),
        _ptr(ref_draft, "ref_draft"), _ptr(tau, "tau", torch.int32, N),
        _ptr(tau_ref, "tau_ref", torch.int32, N),
        _ptr(rollout_len, "rollout_len", torch.float32, nroll),
        _ptr(advantage, "advantage", torch.float32, nroll), _stream(stream))
    _check(code, "aal_accept_reward_noalloc")


def aal_check_device_status(workspace, stream=None) -> int:
    """Synchronise and return (and clear) the workspace's device status code."""
    return int(library().aal_check_device_status(_ptr(workspace, "workspace"), _stream(stream)))


def aal_debug_fail_next_forward(chunk: int, wait_limit_ns: int = 0):
    """Failure-detection test hook: leave one ring copy of the next streamed forward unarmed
    so that its bounded waits run out (see include/aal_debug.h)."""
    library().aal_debug_fail_next_forward(int(chunk), int(wait_limit_ns))


def aal_debug_fused_min_row_bytes(nbytes: int) -> None:
    """Test hook: the shortest row (bytes) aal_loss_fwd_bwd streams with its fused kernels
    (0: every row they take; negative: the default; see include/aal_debug.h)."""
    library().aal_debug_fused_min_row_bytes(int(nbytes))


def aal_debug_solo_windows(N: int, K: int, G: int, S: int) -> int:
    """Test hook: windows per solo CTA that the fused call's launch chooses for N windows of K
    rows, G groups and S spare CTAs (host arithmetic; see include/aal_debug.h)."""
    return int(library().aal_debug_solo_windows(int(N), int(K), int(G), int(S)))
