"""GPU parity of the EAL / WTV forward and backward against the fp64 oracle (through the C ABI)."""

import numpy as np
import pytest
import torch

import oracle
import paper_2609_24150_gb300 as aal
import synth
from tests.parity import LossRun, assert_bands, check_loss, loss_from_eal

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _dev(*ts):
    return [None if t is None else t.to(DEV) for t in ts]


# ------------------------------------------------------------------ tiny workload, all rows

@pytest.mark.parametrize("mode,T,wg,ws", [
    (aal.AAL_GREEDY, 0.0, 1.0, 0.0),
    (aal.AAL_SAMPLING, 1.0, 0.0, 1.0),
    (aal.AAL_BOTH, 1.0, 0.5, 0.5),
    (aal.AAL_BOTH, 0.7, 0.3, 0.7),
    (aal.AAL_SAMPLING, 1.5, 0.0, 1.0),
])
def test_tiny_fp32_all_rows(mode, T, wg, ws):
    target, draft, mask = synth.make_logits("tiny", seed=0)
    t, d = _dev(target, draft)
    run = LossRun(t, d, None, mode, T, wg, ws)
    check_loss(run, t, d, None, mode, T, wg, ws)


@pytest.mark.parametrize("mode", [aal.AAL_GREEDY, aal.AAL_SAMPLING, aal.AAL_BOTH])
def test_tiny_gradient_scaled_by_window_count(mode):
    """dloss = |W| makes the per-element gradients O(q) so the absolute tolerance binds."""
    target, draft, _ = synth.make_logits("tiny", seed=1)
    t, d = _dev(target, draft)
    run = LossRun(t, d, None, mode, 1.0, 0.5, 0.5, dloss=32.0)
    check_loss(run, t, d, None, mode, 1.0, 0.5, 0.5, dloss=32.0)


@pytest.mark.parametrize("V,dtype", [(7, torch.bfloat16), (1001, torch.bfloat16), (4099, torch.float32),
                                     (8, torch.bfloat16), (4096 * 3 + 8, torch.bfloat16),
                                     (1000, torch.bfloat16)])
@pytest.mark.parametrize("K", [1, 3, 8])
def test_ragged_vocab_and_window_sizes(V, dtype, K):
    target, draft, _ = synth.make_logits("tiny", seed=V + K, N=6, K=K, V=V, dtype=dtype)
    mask = torch.ones(6, K, dtype=torch.uint8)
    mask[1, 0] = 0
    if K > 2:
        mask[2, 2] = 0
    t, d, m = _dev(target, draft, mask)
    for mode, T in [(aal.AAL_BOTH, 1.0), (aal.AAL_BOTH, 1.3), (aal.AAL_GREEDY, 0.0)]:
        run = LossRun(t, d, m, mode, T, 0.5, 0.5, dloss=5.0)
        check_loss(run, t, d, m, mode, T, 0.5, 0.5, dloss=5.0)


@pytest.mark.parametrize("V,dtype", [(8, torch.bfloat16), (4096, torch.bfloat16), (4104, torch.bfloat16),
                                     (65544, torch.bfloat16), (100000, torch.bfloat16),
                                     (250000, torch.bfloat16), (40000, torch.float32)])
def test_streamed_row_shapes(V, dtype):
    """Rows of one vector, exactly one chunk, one chunk plus one vector, and many chunks with
    a partial last chunk, through the TMA-streamed forward (row length a multiple of 16 B)."""
    target, draft, _ = synth.make_logits("tiny", seed=V, N=3, K=2, V=V, dtype=dtype)
    draft[1, 1] = target[1, 1]          # an identical row inside a window
    t, d = _dev(target, draft)
    for mode, T in [(aal.AAL_BOTH, 1.0), (aal.AAL_SAMPLING, 0.8), (aal.AAL_BOTH, 1.4)]:
        run = LossRun(t, d, None, mode, T, 0.5, 0.5, dloss=3.0)
        check_loss(run, t, d, None, mode, T, 0.5, 0.5, dloss=3.0)


def test_masked_v32k_sampled_windows():
    """V = 32000 bf16 with 10% of positions masked: sampled windows, loss via the eal outputs."""
    target, draft, mask = synth.make_logits("v32k", seed=0, device=DEV)
    N = target.shape[0]
    kn = oracle.leading_valid_depths(mask.cpu().numpy(), N, 5)
    nvalid = int((kn >= 1).sum())
    rng = np.random.default_rng(0)
    windows = sorted(set([0, N - 1] + list(rng.choice(N, 40, replace=False))))
    for mode, T, wg, ws in [(aal.AAL_GREEDY, 0.0, 1.0, 0.0), (aal.AAL_SAMPLING, 1.0, 0.0, 1.0)]:
        run = LossRun(target, draft, mask, mode, T, wg, ws, dloss=float(nvalid))
        check_loss(run, target, draft, mask, mode, T, wg, ws, dloss=float(nvalid), windows=windows,
                   n_windows_total=nvalid)
        assert_bands()
        implied = loss_from_eal(run, mode, wg, ws, nvalid)
        assert abs(float(run.loss.item()) - implied) <= 1e-5 * abs(implied) + 1e-7
        # masked windows contribute nothing and their rows get exact zeros
        dead = torch.as_tensor(kn == 0, device=DEV)
        assert torch.all(run.grad[dead] == 0)


# ------------------------------------------------------------------ edge cases

def test_no_valid_window():
    target, draft, _ = synth.make_logits("tiny", seed=2, N=5, K=3, V=300, dtype=torch.bfloat16)
    mask = torch.zeros(5, 3, dtype=torch.uint8)
    mask[:, 1:] = 1
    t, d, m = _dev(target, draft, mask)
    run = LossRun(t, d, m, aal.AAL_BOTH, 1.0, 0.5, 0.5)
    assert run.loss.item() == 0.0
    assert torch.all(run.grad == 0)
    assert torch.all(run.eal == 0)


def test_empty_batch():
    d = torch.empty(0, 4, 100, dtype=torch.bfloat16, device=DEV)
    prob = aal.loss_problem(d, aal.AAL_BOTH)
    ws = torch.empty(aal.aal_workspace_size(prob), dtype=torch.uint8, device=DEV)
    loss = torch.full((1,), 3.0, device=DEV)
    aal.aal_loss_fwd(prob, d, d, None, ws, loss)
    aal.aal_loss_bwd(prob, d, d, None, ws, 1.0, d)
    assert loss.item() == 0.0


def test_identical_rows_have_full_overlap_and_zero_wtv_gradient():
    target, _, _ = synth.make_logits("v152k", seed=3, N=4, K=6, V=4000)
    t = target.to(DEV)
    for T in [0.5, 1.0, 1.5]:
        run = LossRun(t, t.clone(), None, aal.AAL_SAMPLING, T, 0.0, 1.0)
        assert torch.all(run.grad == 0)
        np.testing.assert_allclose(run.eal[:, 1].cpu().numpy(), 6.0, rtol=1e-5)


def test_ties_in_target_argmax_take_lowest_index():
    V = 512
    target = torch.zeros(3, 2, V, dtype=torch.bfloat16)
    target[..., 100] = 4.0
    target[..., 300] = 4.0
    target[..., 7] = 4.0
    draft = torch.randn(3, 2, V).to(torch.bfloat16)
    t, d = _dev(target, draft)
    run = LossRun(t, d, None, aal.AAL_GREEDY, 0.0, 1.0, 0.0, dloss=6.0)
    check_loss(run, t, d, None, aal.AAL_GREEDY, 0.0, 1.0, 0.0, dloss=6.0)
    # the +a^g spike of the greedy gradient sits on x* = 7
    g = run.grad.float()
    assert torch.all(g[..., 7] < 0) and torch.all(g[..., 100] > 0)


def test_negative_infinity_logits():
    target, draft, _ = synth.make_logits("tiny", seed=4, N=4, K=3, V=200, dtype=torch.float32)
    target[:, :, 150:] = float("-inf")
    draft[:, :, :20] = float("-inf")
    t, d = _dev(target, draft)
    for mode, T in [(aal.AAL_BOTH, 1.0), (aal.AAL_SAMPLING, 0.6)]:
        run = LossRun(t, d, None, mode, T, 0.5, 0.5, dloss=4.0)
        check_loss(run, t, d, None, mode, T, 0.5, 0.5, dloss=4.0)


def test_peaked_draft_full_greedy_length():
    target, draft, _ = synth.make_logits("tiny", seed=5, N=3, K=5, V=700)
    xs = target.argmax(-1, keepdim=True)
    draft.scatter_(-1, xs, 100.0)
    t, d = _dev(target, draft)
    run = LossRun(t, d, None, aal.AAL_GREEDY, 0.0, 1.0, 0.0)
    np.testing.assert_allclose(run.eal[:, 0].cpu().numpy(), 5.0, rtol=1e-6)


def test_gradient_rows_sum_to_zero():
    target, draft, _ = synth.make_logits("tiny", seed=6, N=8, K=4, V=3000, dtype=torch.float32)
    t, d = _dev(target, draft)
    run = LossRun(t, d, None, aal.AAL_BOTH, 0.9, 0.5, 0.5, dloss=8.0)
    s = run.grad.double().sum(-1).abs().max().item()
    assert s < 1e-5


def test_repeat_calls_are_deterministic():
    target, draft, _ = synth.make_logits("tiny", seed=7, N=64, K=7, V=5000, dtype=torch.bfloat16)
    t, d = _dev(target, draft)
    a = LossRun(t, d, None, aal.AAL_BOTH, 1.0, 0.5, 0.5)
    b = LossRun(t, d, None, aal.AAL_BOTH, 1.0, 0.5, 0.5)
    assert torch.equal(a.loss, b.loss) and torch.equal(a.eal, b.eal) and torch.equal(a.grad, b.grad)


# ------------------------------------------------------------------ full-size workloads

@pytest.fixture(scope="module")
def v128k():
    target, draft, _ = synth.make_logits("v128k", seed=0, device=DEV)
    yield target, draft
    del target, draft
    torch.cuda.empty_cache()


def test_v128k_full_size_sampled_windows(v128k):
    """N=8192, K=7, V=128256 bf16, EAL+WTV 0.5/0.5 at T=1: the benchmark's launch configuration."""
    target, draft = v128k
    N = target.shape[0]
    run = LossRun(target, draft, None, aal.AAL_BOTH, 1.0, 0.5, 0.5, dloss=float(N))
    rng = np.random.default_rng(1)
    windows = sorted(set([0, 1, N - 1] + list(rng.choice(N, 21, replace=False))))
    check_loss(run, target, draft, None, aal.AAL_BOTH, 1.0, 0.5, 0.5, dloss=float(N),
               windows=windows, n_windows_total=N)
    assert_bands()
    implied = loss_from_eal(run, aal.AAL_BOTH, 0.5, 0.5, N)
    assert abs(float(run.loss.item()) - implied) <= 1e-5 * abs(implied)
    # every gradient row is finite and sums to 0 (softmax shift invariance) up to the bf16
    # rounding of its elements: |sum g^| <= 2^-9 sum |g| plus fp32 accumulation error
    for n0 in range(0, N, 512):
        g = run.grad[n0:n0 + 512].double()
        assert torch.isfinite(g).all()
        assert (g.sum(-1).abs() <= 2.0 ** -8 * g.abs().sum(-1) + 1e-9).all()
    del run
    torch.cuda.empty_cache()


@pytest.fixture(scope="module")
def v152k():
    target, draft, _ = synth.make_logits("v152k", seed=0, device=DEV)
    yield target, draft
    del target, draft
    torch.cuda.empty_cache()


@pytest.mark.parametrize("T", [0.5, 1.0, 1.5])
def test_v152k_full_size_temperature_sweep(v152k, T):
    """N=8192, K=6, V=151936, 20% low-overlap rows: WTV at T in {0.5, 1, 1.5}."""
    target, draft = v152k
    N = target.shape[0]
    run = LossRun(target, draft, None, aal.AAL_SAMPLING, T, 0.0, 1.0, dloss=float(N))
    rng = np.random.default_rng(int(T * 10))
    windows = sorted(set([0, N - 1] + list(rng.choice(N, 14, replace=False))))
    check_loss(run, target, draft, None, aal.AAL_SAMPLING, T, 0.0, 1.0, dloss=float(N),
               windows=windows, n_windows_total=N)
    assert_bands()
    # rows whose draft equals the target have an exactly zero WTV gradient, at full size
    for n0 in range(0, N, 512):
        same = (target[n0:n0 + 512] == draft[n0:n0 + 512]).all(-1)
        gmax = run.grad[n0:n0 + 512].abs().amax(-1)
        assert torch.all(gmax[same] == 0)
    del run
    torch.cuda.empty_cache()
