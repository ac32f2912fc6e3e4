"""Seeded synthetic logit workloads for the acceptance-aware losses.

Every workload is a pair of full-vocabulary logit tensors laid out row-major as
[N windows][K window depths][V vocabulary] (the draft ``z_q`` and the frozen
target ``z_p``), plus an optional per-position validity mask [N][K] (1 = valid).
The recipes stand in for the paper's training data (target-generated ShareGPT
continuations truncated to 2048 tokens, Sec. 4.1): the sequence length 2048
fixes T in N = B x T, V = 128256 / 151936 are the vocabulary sizes of the
model families evaluated there, and the logit distributions (Gaussian, Zipf
over a random permutation, heavy-tailed Gumbel, planted peaks, low-overlap rows)
give the range of target/draft overlap that the losses see in training.

Generation is chunked over windows with a fixed chunk size (256 windows), so on
a given device the first ``n`` windows, for ``n`` a multiple of the chunk size,
are the same bytes whether or not the rest is drawn.  Values are drawn in fp32
and rounded once to the storage dtype.
"""

from __future__ import annotations

import dataclasses
from typing import Optional

import torch

WINDOWS_PER_CHUNK = 256


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    N: int
    K: int
    V: int
    dtype: torch.dtype
    recipe: str
    description: str


WORKLOADS = {
    "tiny": Workload(
        "tiny", 32, 4, 1000, torch.float32, "gauss",
        "N=32 (B=2 x 16), K=4, V=1000, fp32; z_p ~ N(0, 3^2), z_q = z_p + N(0, 1)"),
    "v32k": Workload(
        "v32k", 2048, 5, 32000, torch.bfloat16, "peak",
        "N=2048 (B=4 x 512), K=5, V=32000, bf16; z_p ~ N(0, 4^2) plus 8 on one uniform "
        "token per row, z_q = 0.8 z_p + N(0, 1.5^2); 10% of positions masked"),
    "v128k": Workload(
        "v128k", 8192, 7, 128256, torch.bfloat16, "zipf",
        "N=8192 (B=4 x 2048), K=7, V=128256, bf16; z_p = -1.1 ln(rank) + N(0, 0.5^2) with "
        "rank a per-row random permutation of 1..V, z_q = z_p + N(0, 1)"),
    "v152k": Workload(
        "v152k", 8192, 6, 151936, torch.bfloat16, "gumbel",
        "N=8192 (B=4 x 2048), K=6, V=151936, bf16; z_p = 3 Gumbel, z_q = z_p except 20% of "
        "rows replaced by independent 3 Gumbel"),
}

# Reward workload: 64 prompts x 16 rollouts x 256 windows of K=8, V=128256, logits
# drawn per prompt group with the Zipf recipe.
REWARD = dict(prompts=64, rollouts_per_group=16, windows_per_rollout=256, K=8, V=128256,
              dtype=torch.bfloat16)


# Sequence layout (Sec. 3.3): logits stored once per position, [B][seq_len][V], with sliding
# windows of K positions.  The validity mask marks each sequence's prompt (not trained on) and
# the padding after its end: the prompt length is uniform in [prompt_lo, prompt_hi) and the
# sequence ends at a length uniform in [end_lo, seq_len].
@dataclasses.dataclass(frozen=True)
class SeqWorkload:
    name: str
    B: int
    seq_len: int
    K: int
    V: int
    dtype: torch.dtype
    recipe: str
    prompt: tuple
    end_lo: int
    description: str


SEQUENCES = {
    "seq_tiny": SeqWorkload(
        "seq_tiny", 3, 37, 4, 1000, torch.float32, "gauss", (0, 6), 25,
        "B=3 x 37 positions, K=4, V=1000, fp32, gauss recipe; prompts of 0-5 positions, "
        "sequences ending at 25-37"),
    "seq_v128k": SeqWorkload(
        "seq_v128k", 4, 2048, 7, 128256, torch.bfloat16, "zipf", (32, 512), 1024,
        "B=4 x 2048 positions, K=7, V=128256, bf16, zipf recipe; prompts of 32-511 positions, "
        "sequences ending at 1024-2048"),
}

SEQ_ROWS_PER_CHUNK = 2048


def make_seq_logits(name: str, seed: int = 0, device="cpu", B: Optional[int] = None,
                    seq_len: Optional[int] = None, V: Optional[int] = None,
                    dtype: Optional[torch.dtype] = None, masked: bool = True):
    """Draw (target, draft, mask) for a sequence workload: [B][seq_len][V] logits and a
    [B][seq_len] uint8 mask (1 = trained position), or None with ``masked=False``."""
    w = SEQUENCES[name]
    B = w.B if B is None else B
    T = w.seq_len if seq_len is None else seq_len
    V = w.V if V is None else V
    dtype = w.dtype if dtype is None else dtype
    g = _gen(device, seed)
    R = B * T
    target = torch.empty((R, V), dtype=dtype, device=device)
    draft = torch.empty((R, V), dtype=dtype, device=device)
    for r0 in range(0, R, SEQ_ROWS_PER_CHUNK):
        r1 = min(R, r0 + SEQ_ROWS_PER_CHUNK)
        zp, zq = _chunk(w.recipe, r1 - r0, V, g, device)
        target[r0:r1].copy_(zp)
        draft[r0:r1].copy_(zq)
        del zp, zq
    mask = None
    if masked:
        gm = torch.Generator(device="cpu")
        gm.manual_seed(int(seed) + 7919)
        lo, hi = w.prompt
        prompt = torch.randint(min(lo, T), max(min(hi, T), min(lo, T) + 1), (B,), generator=gm)
        end = torch.randint(min(w.end_lo, T), T + 1, (B,), generator=gm)
        t = torch.arange(T)
        mask = ((t[None, :] >= prompt[:, None]) & (t[None, :] < end[:, None])).to(torch.uint8)
        mask = mask.to(device)
    return target.view(B, T, V), draft.view(B, T, V), mask


def workload(name: str) -> Workload:
    return WORKLOADS[name]


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def _gumbel(shape, g, device):
    u = torch.rand(shape, generator=g, device=device, dtype=torch.float32)
    u = u.clamp_(min=1e-12, max=1.0 - 1e-7)
    return -torch.log(-torch.log(u))


def _zipf_rows(rows, V, g, device):
    # rank = 1 + pi(v) for a uniformly random permutation pi of the row
    perm = torch.argsort(torch.rand((rows, V), generator=g, device=device), dim=1)
    rank = torch.empty((rows, V), device=device, dtype=torch.float32)
    rank.scatter_(1, perm, torch.arange(1, V + 1, device=device, dtype=torch.float32)
                  .expand(rows, V).contiguous())
    del perm
    return -1.1 * torch.log(rank) + 0.5 * torch.randn((rows, V), generator=g, device=device)


def _chunk(recipe, rows, V, g, device):
    """One chunk of (target, draft) fp32 logits, ``rows`` logit rows each."""
    if recipe == "gauss":
        zp = 3.0 * torch.randn((rows, V), generator=g, device=device)
        zq = zp + torch.randn((rows, V), generator=g, device=device)
    elif recipe == "peak":
        zp = 4.0 * torch.randn((rows, V), generator=g, device=device)
        tok = torch.randint(0, V, (rows, 1), generator=g, device=device)
        zp.scatter_add_(1, tok, torch.full((rows, 1), 8.0, device=device))
        zq = 0.8 * zp + 1.5 * torch.randn((rows, V), generator=g, device=device)
    elif recipe == "zipf":
        zp = _zipf_rows(rows, V, g, device)
        zq = zp + torch.randn((rows, V), generator=g, device=device)
    elif recipe == "gumbel":
        zp = 3.0 * _gumbel((rows, V), g, device)
        other = 3.0 * _gumbel((rows, V), g, device)
        swap = torch.rand((rows, 1), generator=g, device=device) < 0.2
        zq = torch.where(swap, other, zp)
    else:
        raise ValueError(recipe)
    return zp, zq


def make_logits(name: str, seed: int = 0, device="cpu", n_windows: Optional[int] = None,
                N: Optional[int] = None, K: Optional[int] = None, V: Optional[int] = None,
                dtype: Optional[torch.dtype] = None, mask_rate: Optional[float] = None):
    """Draw (target, draft, mask) for a named workload.

    ``n_windows`` draws only the first windows of the workload (same bytes as the
    full draw); ``N``/``K``/``V``/``dtype`` override the shape for edge-case tests.
    Returns ``target [N,K,V]``, ``draft [N,K,V]`` and ``mask [N,K]`` (uint8, 1 =
    valid) or ``None`` when the workload masks nothing.
    """
    w = WORKLOADS[name]
    N_full = w.N if N is None else N
    K = w.K if K is None else K
    V = w.V if V is None else V
    dtype = w.dtype if dtype is None else dtype
    N = N_full if n_windows is None else min(N_full, n_windows)
    g = _gen(device, seed)
    target = torch.empty((N, K, V), dtype=dtype, device=device)
    draft = torch.empty((N, K, V), dtype=dtype, device=device)
    for n0 in range(0, N, WINDOWS_PER_CHUNK):
        n1 = min(N, n0 + WINDOWS_PER_CHUNK)
        zp, zq = _chunk(w.recipe, (n1 - n0) * K, V, g, device)
        target[n0:n1].copy_(zp.view(n1 - n0, K, V))
        draft[n0:n1].copy_(zq.view(n1 - n0, K, V))
        del zp, zq
    rate = (0.1 if w.recipe == "peak" else 0.0) if mask_rate is None else mask_rate
    mask = None
    if rate > 0.0:
        gm = _gen(device, seed + 7919)
        mask = (torch.rand((N_full, K), generator=gm, device=device) >= rate).to(torch.uint8)
        mask = mask[:N].contiguous()
    return target, draft, mask


def make_reward_logits(group: int, seed: int = 0, device="cpu", with_ref: bool = False,
                       windows_per_rollout: Optional[int] = None,
                       rollouts_per_group: Optional[int] = None, K: Optional[int] = None,
                       V: Optional[int] = None, dtype: Optional[torch.dtype] = None,
                       ref_from_draft: Optional[float] = None):
    """Draw one prompt group of the reward workload: (target, draft, ref_draft | None).

    Rows are [rollouts_per_group * windows_per_rollout][K][V]; the group is drawn
    from its own generator seeded by (seed, group), so groups can be streamed one
    at a time. ``ref_draft`` (a frozen earlier draft) is the target plus its own
    independent N(0, 1) noise, or, with ``ref_from_draft = s``, the draft plus N(0, s^2)
    noise: a snapshot of the draft a little way back in training, as the GRPO stage's
    reference policy is.
    """
    wpr = REWARD["windows_per_rollout"] if windows_per_rollout is None else windows_per_rollout
    rpg = REWARD["rollouts_per_group"] if rollouts_per_group is None else rollouts_per_group
    K = REWARD["K"] if K is None else K
    V = REWARD["V"] if V is None else V
    dtype = REWARD["dtype"] if dtype is None else dtype
    N = wpr * rpg
    g = _gen(device, seed * 65536 + group + 1)
    target = torch.empty((N, K, V), dtype=dtype, device=device)
    draft = torch.empty((N, K, V), dtype=dtype, device=device)
    ref = torch.empty((N, K, V), dtype=dtype, device=device) if with_ref else None
    for n0 in range(0, N, WINDOWS_PER_CHUNK):
        n1 = min(N, n0 + WINDOWS_PER_CHUNK)
        rows = (n1 - n0) * K
        zp = _zipf_rows(rows, V, g, device)
        target[n0:n1].copy_(zp.view(n1 - n0, K, V))
        draft[n0:n1].copy_((zp + torch.randn((rows, V), generator=g, device=device))
                           .view(n1 - n0, K, V))
        if with_ref:
            if ref_from_draft is None:
                ref[n0:n1].copy_((zp + torch.randn((rows, V), generator=g, device=device))
                                 .view(n1 - n0, K, V))
            else:
                zq = draft[n0:n1].view(rows, V).float()
                ref[n0:n1].copy_((zq + ref_from_draft * torch.randn((rows, V), generator=g, device=device))
                                 .view(n1 - n0, K, V))
                del zq
        del zp
    return target, draft, ref


def bytes_per_tensor(N: int, K: int, V: int, dtype: torch.dtype) -> int:
    return N * K * V * (torch.finfo(dtype).bits // 8)


def human_gb(nbytes: int) -> str:
    return f"{nbytes / 1e9:.2f} GB"


__all__ = ["Workload", "WORKLOADS", "REWARD", "SeqWorkload", "SEQUENCES", "workload", "make_logits",
           "make_reward_logits", "make_seq_logits", "bytes_per_tensor", "human_gb"]
