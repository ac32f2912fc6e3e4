"""Oracle for the acceptance-aware draft-training losses -- TEST INFRASTRUCTURE ONLY.

A plain, slow, fp64 CPU restatement of what the paper defines: the per-position
acceptance probabilities under greedy and sampling verification (Sec. 2.3,
Eqs. acc_greedy / acc_sample), the speculative-window expected accepted length
(Sec. 3.1, Eq. eal_generic), the EAL and WTV losses (Eqs. loss_eal / loss_tv)
with their gradient with respect to the draft logits, over independent windows and
over whole sequences (Sec. 3.3), the forward-KL anchor of the combined objectives
(Sec. 4.1), the GRPO stage's clipped policy-ratio surrogate (Sec. 3.4), and its
simulated acceptance length, debiased reward and group-normalised advantage
(Sec. 3.4).  Every function computes its definition directly, with numpy in
float64, so that a reader can check it against the paper by eye; nothing here
is blocked, fused or reordered for speed.

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline leg
may import this package.  The product library never calls it, and it shares no
code with the CUDA path: the two meet only in the seeded inputs of ``synth``.

Parity status: every function is pinned by the ``-m "not gpu"`` tests to facts
the paper or mathematics fixes (brute-force enumeration of speculative
verification, the gamma = 3 worked example, closed forms, finite differences,
Monte Carlo, and for the counter-based generator the independent cuRAND host
implementation).  No function here is parity-unpinned.
"""

from .losses import (  # noqa: F401
    MODE_BOTH,
    MODE_GREEDY,
    MODE_SAMPLING,
    acceptance_greedy,
    acceptance_sampling,
    argmax_lowest,
    as_f64,
    expected_length,
    expected_length_partials,
    leading_valid_depths,
    log_softmax,
    loss_backward,
    loss_forward,
    row_acceptances,
)
from .reward import (  # noqa: F401
    accept_reward,
    debiased_reward,
    greedy_trajectory,
    group_advantages,
    REWARD_SAMPLED_DRAFT,
    rollout_lengths,
    sampled_trajectory,
    sampling_accepts,
    sampling_accepts_at,
    simulated_accept_length,
)
from .philox import gumbel_uniforms, philox4x32_10, uniform01  # noqa: F401
from .sequence import (  # noqa: F401
    gather_windows,
    seq_loss_backward,
    seq_loss_forward,
    seq_objective_backward,
    seq_objective_forward,
)
from .grpo import grpo_backward, grpo_forward, policy_log_ratio, trajectory_log_probs  # noqa: F401
from .anchor import (  # noqa: F401
    MODE_KL,
    MODE_TV,
    anchor_backward,
    anchor_forward,
    kl_divergence,
    objective_backward,
    objective_forward,
    total_variation,
    tv_backward,
    tv_forward,
)
