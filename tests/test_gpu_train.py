"""GPU parity of the training-time pathway's forward (Sec. 3.3, Eqs. 5-9)
through the C ABI against the CPU oracle on the same seeded inputs.

Comparison rules:
  * the hard rollout of sp_select_train is sp_select's, bit for bit (same
    decisions from the same kernel code);
  * scores s (Eq. 6) and soft counts Kbar (Eq. 7): the oracle is replayed along
    the GPU's rollout (teacher forcing, stage-local) and fed the same candidate
    memory; |gpu - oracle| <= S_RTOL |oracle| + S_ATOL.  The GPU's logits differ
    from the oracle's by the fp32 rounding of the folded decoder (the inference
    tests allow 2e-4 on per-round gaps); a logit error d moves p_t(j) by at most
    2 d / tau relative, which bounds the relative error of every sum of Eqs. 6-7;
  * alpha (Eq. 8) from the GPU's own s / Kbar: within ALPHA_ATOL of the
    oracle's Sinkhorn solution (fp32 sigmoids around an fp32 threshold);
  * the gate (Eq. 9): bf16 output within one bf16 rounding (2^-8 relative) of
    the fp64 value on the same bf16 inputs; alpha = 1 / 0 exact.
"""
import numpy as np
import pytest

import _parity as PT
from oracle import core as O
from paper_2609_13804_gb300 import synth as S

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

DEV = "cuda"
S_RTOL = 2e-3
S_ATOL = 1e-6
ALPHA_ATOL = 2e-5


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_13804_gb300 import binding
    binding.lib()
    return binding


def np_(t):
    return t.float().cpu().numpy() if t.dtype == torch.bfloat16 else t.cpu().numpy()


def _train_case(B, w, *, tau, beta, scale=1.0, targets=None, sample=None, mean_target=None):
    """Runs sp_select and sp_select_train on the same inputs; replays the oracle
    along the GPU rollout for the episodes in `sample` (all if None)."""
    sel = S.make_selector_weights(w, ln_affine=True)
    if scale != 1.0:
        PT.scale_decoder(sel, scale)
    H = S.make_memory(w)
    eps_list = PT.episodes(w.n_vis, w.group_size)
    if targets is None:
        targets = S.uniform_int(w.seed, "targets", 0, w.k_max + 1, len(eps_list))
    biases = PT.calibrate_biases(H, w.n_vis, sel, k_max=w.k_max, g=1, group_size=w.group_size, targets=targets,
                                 mean_target=mean_target)
    s = w.selector
    shape = S.SelectorShape(D=s.D, D_text=s.D_text, h=s.h, n_enc_layers=0)
    selector = B.Selector(shape, sel, DEV)
    Hd, bd = B.dev_f32(H, DEV), B.dev_f32(biases, DEV)
    ref = B.sp_select(selector, w.n_vis, w.n_txt, H=Hd, stop_bias=bd, group_size=w.group_size, g=1, k_max=w.k_max)
    got = B.sp_select(selector, w.n_vis, w.n_txt, H=Hd, stop_bias=bd, group_size=w.group_size, g=1, k_max=w.k_max,
                      train=(tau, beta))
    torch.cuda.synchronize()
    assert int(got["err"].item()) == 0
    for k in ("idx", "count", "order", "ep_count", "rounds", "margin", "gap"):
        np.testing.assert_array_equal(np_(got[k]), np_(ref[k]), err_msg=k)
    g = {k: np_(got[k]) for k in ("order", "ep_count", "rounds", "score", "kbar")}
    offs = np.concatenate([[0], np.cumsum(w.n_vis)])
    worst = 0.0
    for e, (b, c0, n) in enumerate(eps_list):
        if sample is not None and e not in sample:
            continue
        cnt = int(g["ep_count"][e])
        order = [int(x) for x in g["order"][e][:cnt]]
        stopped = int(g["rounds"][e]) > cnt
        r = O.trajectory_episode(H[offs[b] + c0: offs[b] + c0 + n].astype(np.float64), sel, k_max=w.k_max,
                                 tau=tau, beta=beta, stop_bias=float(biases[e]), force=order, force_stop=stopped)
        assert r["rounds"] == int(g["rounds"][e])
        gs = g["score"][offs[b] + c0: offs[b] + c0 + n].astype(np.float64)
        err = np.abs(gs - r["s"])
        assert np.all(err <= S_RTOL * np.abs(r["s"]) + S_ATOL), (e, err.max())
        assert abs(g["kbar"][e] - r["kbar"]) <= S_RTOL * abs(r["kbar"]) + S_ATOL, (e, g["kbar"][e], r["kbar"])
        worst = max(worst, float(np.max(err / (np.abs(r["s"]) + 1e-3))))
    print("worst relative score error", worst)
    selector.close()
    return g, biases, H


def test_train_tiny_ragged(B):
    w = S.tiny_workload(31, [37, 5, 130, 1, 64], [3, 0, 2, 1, 4], D=128, h=128, k_max=12)
    _train_case(B, w, tau=1.0, beta=0.9, scale=4.0)


@pytest.mark.parametrize("tau,beta", [(0.25, 1.0), (3.0, 0.7)])
def test_train_tiny_groups_and_temperatures(B, tau, beta):
    w = S.tiny_workload(32, [300, 77, 128], [2, 2, 2], D=128, h=256, k_max=20, group_size=128)
    g, _, _ = _train_case(B, w, tau=tau, beta=beta, scale=4.0)
    if beta == 1.0:  # every p_t sums to one: sum_i s_i = Kbar per episode
        offs = np.concatenate([[0], np.cumsum(w.n_vis)])
        for e, (b, c0, n) in enumerate(PT.episodes(w.n_vis, w.group_size)):
            tot = float(np.sum(g["score"][offs[b] + c0: offs[b] + c0 + n], dtype=np.float64))
            assert abs(tot - g["kbar"][e]) <= 1e-5 * max(1.0, g["kbar"][e])


def test_train_stop_extremes(B):
    """STOP wins at once (Kbar from one step), the cap ends a rollout, and an
    exhausted episode ends with a STOP-only step that adds nothing."""
    w = S.tiny_workload(33, [9, 20, 3], [1, 1, 1], D=128, h=128, k_max=8)
    g, _, _ = _train_case(B, w, tau=0.5, beta=0.9, scale=4.0, targets=[0, 8, 3])
    assert int(g["ep_count"][0]) == 0 and int(g["rounds"][0]) == 1
    assert int(g["rounds"][1]) == 8 and int(g["rounds"][2]) == 4


def test_train_llava15_b16_sampled(B):
    """16 x 576 candidates, h = 512, cap 192, the benchmark's kept counts; the
    oracle replays 4 of the 16 episodes (the longest among them)."""
    w = S.llava15_7b_b16()
    t = S.target_counts(w)
    longest = int(np.argmax(t))
    _train_case(B, w, tau=1.0, beta=0.99, targets=t, mean_target=w.target_mean_k,
                sample={0, 5, 11, longest})


# ------------------------------------------------------------------ Eq. 8

def _topk_case(B, n_vis, group_size, seed, tau):
    E = B.sp_num_episodes(n_vis, group_size)
    s = S.normal(seed, "s", (sum(n_vis),)) ** 2 * 0.1  # non-negative, like Eq. 6 scores
    kb = np.abs(S.normal(seed, "kbar", (E,))) * 30.0
    r = B.sp_soft_topk(n_vis, score=B.dev_f32(s, DEV), kbar=B.dev_f32(kb, DEV), tau=tau, group_size=group_size)
    torch.cuda.synchronize()
    alpha, k = np_(r["alpha"]), float(r["k"].item())
    offs = np.concatenate([[0], np.cumsum(n_vis)])
    img = [kb[e0:e1].astype(np.float64).sum() for e0, e1 in _ep_ranges(n_vis, group_size)]
    k_ref = float(np.mean(img))
    assert abs(k - k_ref) <= 1e-5 * k_ref
    for b, n in enumerate(n_vis):
        want = O.soft_topk(s[offs[b]:offs[b + 1]].astype(np.float64), min(max(k_ref, 0.0), n), tau)
        np.testing.assert_allclose(alpha[offs[b]:offs[b + 1]], want, atol=ALPHA_ATOL, err_msg=f"image {b}")
    return alpha, k


def _ep_ranges(n_vis, group_size):
    out, e = [], 0
    for n in n_vis:
        ne = (n + group_size - 1) // group_size if group_size > 0 else 1
        out.append((e, e + ne))
        e += ne
    return out


def test_soft_topk_llava_batch(B):
    _topk_case(B, [576] * 16, 0, 41, 0.05)


def test_soft_topk_groups_ragged_and_clamped(B):
    # image 1 (5 tokens) has k above its size: every token kept (alpha = 1)
    alpha, k = _topk_case(B, [300, 5, 1000, 64], 128, 42, 0.1)
    assert k > 5
    np.testing.assert_array_equal(alpha[300:305], 1.0)


def test_soft_topk_zero_count(B):
    r = B.sp_soft_topk([10, 20], score=B.dev_f32(np.linspace(0, 1, 30), DEV),
                       kbar=B.dev_f32(np.zeros(2), DEV), tau=0.1)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(np_(r["alpha"]), 0.0)


# ------------------------------------------------------------------ Eq. 9

@pytest.mark.parametrize("rows,D", [(1000, 1024), (7, 4096), (1, 8)])
def test_vp_gate(B, rows, D):
    X = S.bf16_round(S.normal(51, "X", (rows, D)))
    Nz = S.bf16_round(S.normal(51, "eps", (rows, D)))
    a = np.abs(S.normal(51, "a", (rows,))) % 1.0
    a[0] = 1.0
    if rows > 1:
        a[1] = 0.0
    Xd, Nd = B.dev_bf16(X, DEV), B.dev_bf16(Nz, DEV)
    out = B.sp_vp_gate(X=Xd, noise=Nd, alpha=B.dev_f32(a, DEV))
    torch.cuda.synchronize()
    got = np_(out)
    ref = O.vp_gate(X.astype(np.float64), a, Nz.astype(np.float64))
    # one bf16 rounding of the result plus the fp32 rounding of its two terms
    terms = np.sqrt(a)[:, None] * np.abs(X) + np.sqrt(1 - a)[:, None] * np.abs(Nz)
    assert np.all(np.abs(got - ref) <= 2.0 ** -8 * np.abs(ref) + 2.0 ** -22 * terms)
    np.testing.assert_array_equal(got[0], X[0])
    if rows > 1:
        np.testing.assert_array_equal(got[1], Nz[1])
