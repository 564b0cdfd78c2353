"""Pins of the oracle's training-time pathway (Sec. 3.3, Eqs. 5-9) against
closed forms, invariants, brute force and limits.  No GPU, no CUDA library."""
import math

import numpy as np
import pytest

from oracle import core as O
from paper_2609_13804_gb300 import synth as S


def _scaled_selector(seed, N=14, D=24, h=16, scale=0.3):
    w = S.tiny_workload(seed, [N], [3], D=D, h=h)
    sel = S.make_selector_weights(w, ln_affine=True)
    for n in ("W_in", "Wq_s", "Wk_s", "Wv_s", "Wo_s", "Wq_p", "Wk_p", "s_start", "s_stop"):
        sel[n] = (sel[n] / 0.02 * scale / math.sqrt(sel[n].shape[-1])).astype(np.float32)
    return sel, S.make_memory(w).astype(np.float64)


# ---------------------------------------------------------------- Eqs. 5-7

@pytest.mark.parametrize("c,beta,T,n", [(0.1, 0.9, 7, 5), (0.35, 1.0, 12, 3), (0.02, 0.97, 40, 9)])
def test_aggregate_constant_stop_probability_closed_forms(c, beta, T, n):
    """p_t(STOP) = c and the rest spread evenly over n visual slots at every
    step: A_t = (1-c)^(t-1), Kbar and s_i are finite geometric series."""
    P = np.zeros((T, n + 1))
    P[:, :n] = (1 - c) / n
    P[:, n] = c
    r = O.trajectory_aggregate(P, beta)
    q = 1 - c
    np.testing.assert_allclose(r["alive"], q ** np.arange(T), rtol=1e-13)
    np.testing.assert_allclose(r["kbar"], q * (1 - q ** T) / c, rtol=1e-13)
    x = beta * q
    geo = beta * (1 - x ** T) / (1 - x) if x != 1 else beta * T
    np.testing.assert_allclose(r["s"], np.full(n, q / n * geo), rtol=1e-12)


def test_aggregate_one_hot_steps():
    """Hard (one-hot) distributions: A stays 1 until STOP is certain, each chosen
    token scores beta^t of its step, Kbar counts the non-STOP steps."""
    P = np.zeros((4, 6))
    for t, j in enumerate([2, 0, 4, 5]):  # the last step is STOP (slot 5)
        P[t, j] = 1.0
    r = O.trajectory_aggregate(P, 0.5)
    np.testing.assert_array_equal(r["alive"], [1, 1, 1, 1])
    assert r["kbar"] == 3
    np.testing.assert_allclose(r["s"], [0.25, 0, 0.5, 0, 0.125])


@pytest.mark.parametrize("seed", range(6))
def test_scores_sum_to_soft_count_without_discount(seed):
    """Every p_t sums to one over the available tokens and STOP, so at beta = 1
    the scores of Eq. 6 add up to the soft count of Eq. 7."""
    sel, H = _scaled_selector(400 + seed, N=12)
    for tau in (0.5, 1.0, 3.0):
        r = O.trajectory_episode(H, sel, k_max=9, tau=tau, beta=1.0, stop_bias=-0.2)
        assert abs(r["s"].sum() - r["kbar"]) < 1e-12
        assert np.all(r["s"] >= 0) and 0 <= r["kbar"] <= r["rounds"]
        np.testing.assert_allclose(r["P"].sum(axis=1), 1.0, atol=1e-14)


@pytest.mark.parametrize("seed", range(8))
def test_rollout_is_the_inference_selection(seed):
    """The hard rollout under the distributions is Eq. 4's inference rollout
    (g = 1): same order, count, stop flag and evaluated rounds."""
    sel, H = _scaled_selector(500 + seed, N=10 + seed % 4)
    for bias in (-1e9, -0.3, 0.0, 0.4):
        for k_max in (3, 8, 20):
            a = O.select_episode(H, sel, k_max=k_max, g=1, stop_bias=bias)
            b = O.trajectory_episode(H, sel, k_max=k_max, tau=0.7, beta=0.9, stop_bias=bias)
            assert (a["order"], a["stopped"], a["rounds"]) == (b["order"], b["stopped"], b["rounds"])


@pytest.mark.parametrize("seed", range(4))
def test_scratch_equals_incremental_and_forcing_own_rollout_is_identity(seed):
    sel, H = _scaled_selector(600 + seed, N=11)
    a = O.trajectory_episode(H, sel, k_max=7, tau=0.5, beta=0.95, stop_bias=-0.1)
    b = O.trajectory_episode(H, sel, k_max=7, tau=0.5, beta=0.95, stop_bias=-0.1, mode="scratch")
    c = O.trajectory_episode(H, sel, k_max=7, tau=0.5, beta=0.95, stop_bias=-0.1, force=a["order"],
                             force_stop=a["stopped"])
    for r in (b, c):
        assert r["order"] == a["order"] and r["rounds"] == a["rounds"]
        np.testing.assert_allclose(r["s"], a["s"], atol=1e-12)
        assert abs(r["kbar"] - a["kbar"]) < 1e-12


def test_forcing_another_rollout_changes_the_history():
    """Teacher forcing replays the given actions (the history follows them)."""
    sel, H = _scaled_selector(650, N=9)
    a = O.trajectory_episode(H, sel, k_max=4, tau=1.0, beta=1.0, stop_bias=-1e9)
    other = [j for j in range(9) if j not in a["order"]][:4]
    r = O.trajectory_episode(H, sel, k_max=4, tau=1.0, beta=1.0, stop_bias=-1e9, force=other, force_stop=False)
    assert r["order"] == other and r["rounds"] == 4
    assert not np.allclose(r["P"][1:], a["P"][1:])


@pytest.mark.parametrize("seed", range(6))
def test_zero_temperature_limit_counts_the_hard_selection(seed):
    """tau -> 0: p_t becomes the one-hot of the argmax, so A stays 1, Kbar is the
    hard count and each kept token scores beta^t of the step that took it."""
    sel, H = _scaled_selector(700 + seed, N=12)
    for bias in (-0.2, 0.3, -1e9):
        base = O.select_episode(H, sel, k_max=8, g=1, stop_bias=bias)
        if min(base["margin"]) < 1e-2:
            continue  # a near tie would not be one-hot at this temperature
        r = O.trajectory_episode(H, sel, k_max=8, tau=1e-5, beta=0.8, stop_bias=bias)
        assert abs(r["kbar"] - r["count"]) < 1e-9
        want = np.zeros(H.shape[0])
        for t, j in enumerate(r["order"], start=1):
            want[j] = 0.8 ** t
        np.testing.assert_allclose(r["s"], want, atol=1e-9)


# ---------------------------------------------------------------- Eq. 8

def _sigmoid_threshold(s, k, tau):
    """Closed form of the two-anchor entropic transport: the plan's row ratio is
    exp((2 s_i - 1 + g_2 - g_1) / tau), so alpha_i = sigmoid(2 (s_i - theta) / tau)
    with theta fixed by Sum alpha = k.  theta by plain bisection."""
    s = np.asarray(s, np.float64)
    lo, hi = s.min() - 50 * tau, s.max() + 50 * tau
    f = lambda th: np.sum(1 / (1 + np.exp(-2 * (s - th) / tau))) - k  # noqa: E731
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if f(mid) > 0:
            lo = mid
        else:
            hi = mid
    th = 0.5 * (lo + hi)
    return 1 / (1 + np.exp(-2 * (s - th) / tau))


@pytest.mark.parametrize("n,k,tau", [(50, 1, 0.05), (50, 7.5, 0.2), (50, 25, 0.1), (50, 49, 0.3), (300, 40.2, 0.02)])
def test_soft_topk_equals_its_closed_form(n, k, tau):
    s = np.random.default_rng(n + int(10 * k)).gamma(1.0, 0.2, n)
    a = O.soft_topk(s, k, tau)
    np.testing.assert_allclose(a, _sigmoid_threshold(s, k, tau), atol=1e-10)
    assert abs(a.sum() - k) < 1e-9
    assert np.all((a >= 0) & (a <= 1 + 1e-12))
    order = np.argsort(s)
    assert np.all(np.diff(a[order]) >= -1e-12)  # monotone in the score
    perm = np.random.default_rng(1).permutation(n)
    np.testing.assert_allclose(O.soft_topk(s[perm], k, tau), a[perm], atol=1e-10)


def test_soft_topk_two_tokens_is_logistic():
    for s1, s2, tau in [(0.3, 0.1, 0.1), (0.0, 1.0, 0.5), (2.0, 2.0, 0.3)]:
        a = O.soft_topk([s1, s2], 1, tau)
        want = 1 / (1 + math.exp(-(s1 - s2) / tau))
        np.testing.assert_allclose(a, [want, 1 - want], atol=1e-12)


def test_soft_topk_limits():
    # three clearly leading scores: well below their lead the transport sends
    # those to the "kept" anchor (error ~ exp(-lead / tau); Sinkhorn converges
    # slowly here, so the set is small)
    s8 = np.array([1.0, 0.02, 0.95, 0.0, 0.05, 0.97, 0.03, 0.01])
    np.testing.assert_allclose(O.soft_topk(s8, 3, 0.1), (s8 > 0.5).astype(float), atol=2e-4)
    s = np.random.default_rng(3).uniform(0, 1, 40)
    np.testing.assert_array_equal(O.soft_topk(s, 0, 0.1), np.zeros(40))
    np.testing.assert_array_equal(O.soft_topk(s, 40, 0.1), np.ones(40))
    a = O.soft_topk(s, 12, 1e3)  # very soft: every token near k / n
    np.testing.assert_allclose(a, 12 / 40, atol=2e-3)


# ---------------------------------------------------------------- Eq. 9

def test_vp_gate_ends_and_variance():
    rng = np.random.default_rng(4)
    x = rng.standard_normal((6, 8))
    e = rng.standard_normal((6, 8))
    a = np.array([1.0, 0.0, 0.25, 0.5, 0.9, 0.01])
    g = O.vp_gate(x, a, e)
    np.testing.assert_array_equal(g[0], x[0])
    np.testing.assert_array_equal(g[1], e[1])
    # unit-variance x and independent unit-variance noise stay unit variance
    X = rng.standard_normal((4, 250_000))
    E = rng.standard_normal((4, 250_000))
    G = O.vp_gate(X, np.array([0.1, 0.4, 0.7, 0.95]), E)
    np.testing.assert_allclose(G.var(axis=1), 1.0, atol=1.5e-2)
    np.testing.assert_allclose(np.mean(G * X, axis=1), np.sqrt([0.1, 0.4, 0.7, 0.95]), atol=1.5e-2)


def test_train_forward_batch_composition():
    """k is the detached batch mean of the images' soft counts; each image's
    alpha sums to it; candidate groups add their soft counts per image."""
    w = S.tiny_workload(11, [10, 7], [3, 2], D=24, h=16)
    sel = S.make_selector_weights(w, ln_affine=True)
    for n in ("W_in", "Wq_s", "Wk_s", "Wv_s", "Wo_s", "Wq_p", "Wk_p", "s_start", "s_stop"):
        sel[n] = (sel[n] / 0.02 * 0.3 / math.sqrt(sel[n].shape[-1])).astype(np.float32)
    H = S.make_memory(w).astype(np.float64)
    r = O.train_forward(H, [10, 7], sel, k_max=5, group_size=4, tau=0.8, beta=0.9, topk_tau=0.05,
                        stop_bias=[0.0] * 5)
    assert len(r["kbar"]) == 3 + 2
    np.testing.assert_allclose(r["kbar_image"], [r["kbar"][:3].sum(), r["kbar"][3:].sum()], rtol=1e-14)
    assert abs(r["k"] - r["kbar_image"].mean()) < 1e-14
    assert abs(r["alpha"][:10].sum() - min(r["k"], 10)) < 1e-8
    assert abs(r["alpha"][10:].sum() - min(r["k"], 7)) < 1e-8
    # group 2 of image 0 is an independent episode over candidates 4..7
    g2 = O.trajectory_episode(H[4:8], sel, k_max=5, tau=0.8, beta=0.9, stop_bias=0.0)
    np.testing.assert_allclose(r["s"][4:8], g2["s"], atol=1e-14)
