"""The selection comparison rule of the GPU parity tests, exercised on the CPU
with the oracle standing in for the GPU: an exact trajectory passes, a swap of
two near-tied candidates passes through the teacher-forced continuation, and a
decision far from the oracle's best fails."""
import numpy as np
import pytest

import _parity as PT
from oracle import core as O
from paper_2609_13804_gb300 import synth as S


def _case(twin_gap):
    w = S.tiny_workload(77, [40, 25], [1, 1], D=32, h=32, k_max=10)
    sel = PT.scale_decoder(S.make_selector_weights(w, ln_affine=True), 3.0)
    H = S.make_memory(w).astype(np.float64)
    free = O.select_episode(H[:40], sel, k_max=10, stop_bias=-1e30)
    a = free["order"][3]
    b = [j for j in range(40) if j not in free["order"]][0]
    H[b] = H[a] * (1.0 + twin_gap)  # a twin of the fourth pick, slightly scaled
    biases = np.array([-1e30, 0.0])
    return w, sel, H, biases, a, b


def _as_gpu(images, k_max, k_cap):
    eps = [ep for img in images for ep in img["episodes"]]
    order = np.full((len(eps), k_max), -1, np.int64)
    for e, ep in enumerate(eps):
        order[e, :ep["count"]] = ep["order"]
    idx = np.full((len(images), k_cap), -1, np.int64)
    for b, img in enumerate(images):
        idx[b, :img["count"]] = img["idx"]
    return {"order": order, "ep_count": np.array([ep["count"] for ep in eps]),
            "rounds": np.array([ep["rounds"] for ep in eps]),
            "gap": np.array([np.pad(np.asarray(ep["gap"], float), (0, k_max + 1 - len(ep["gap"])))
                             for ep in eps]),
            "idx": idx, "count": np.array([img["count"] for img in images])}


def _compare(w, sel, H, biases, gpu):
    images = PT.oracle_select(H, w.n_vis, sel, k_max=w.k_max, g=1, group_size=0, biases=biases)
    replay, eps_list = PT.replayer(H, w.n_vis, sel, k_max=w.k_max, g=1, group_size=0, biases=biases)
    report = []
    near = PT.compare_selection(gpu, images, g=1, report=report, replay=replay, episodes=eps_list)
    return near, report


def test_exact_trajectory_passes():
    w, sel, H, biases, _, _ = _case(0.3)
    images = PT.oracle_select(H, w.n_vis, sel, k_max=w.k_max, g=1, group_size=0, biases=biases)
    near, _ = _compare(w, sel, H, biases, _as_gpu(images, w.k_max, 40))
    assert near == 0


def _swapped_gpu(w, sel, H, biases, a, b):
    """The oracle's result with the near-tied twin taken instead of a (and the
    rest of the episode teacher-forced from there, as another implementation
    that resolved the tie the other way would continue)."""
    images = PT.oracle_select(H, w.n_vis, sel, k_max=w.k_max, g=1, group_size=0, biases=biases)
    ep = images[0]["episodes"][0]
    k = min(ep["order"].index(a), ep["order"].index(b))
    other = b if ep["order"][k] == a else a
    order = list(ep["order"][:k]) + [other]
    while len(order) < w.k_max:  # continue greedily along the swapped history
        taken = set(order)
        cand = [j for j in range(40) if j not in taken]
        best = max(cand, key=lambda j: (_logit_after(H, sel, order, j), -j))
        order.append(best)
    gpu = _as_gpu(images, w.k_max, 40)
    gpu["order"][0, :len(order)] = order
    gpu["idx"][0, :len(order)] = sorted(order)
    return gpu, order


def _logit_after(H, sel, order, j):
    M = np.concatenate([H[:40], sel["s_stop"][None].astype(np.float64)])
    hist = [sel["s_start"].astype(np.float64)] + [M[i] for i in order]
    return O.pointer_logits_from_scratch(np.stack(hist), M, sel, 1e-5)[j]


def test_near_tie_swap_passes_through_teacher_forcing():
    w, sel, H, biases, a, b = _case(1e-9)
    gpu, order = _swapped_gpu(w, sel, H, biases, a, b)
    # the forced replay has the same gaps as the oracle's free run only up to the swap
    near, report = _compare(w, sel, H, biases, gpu | {"gap": _forced_gaps(w, sel, H, biases, order, gpu)})
    assert near == 1 and "teacher-forced" in report[0]


def _forced_gaps(w, sel, H, biases, order, gpu):
    f = O.select_episode(H[:40], sel, k_max=w.k_max, g=1, stop_bias=-1e30, force=order)
    g = gpu["gap"].copy()
    g[0, :len(f["gap"])] = f["gap"]
    return g


def test_decision_far_from_the_best_fails():
    w, sel, H, biases, a, b = _case(1e-9)
    gpu, order = _swapped_gpu(w, sel, H, biases, a, b)
    gpu["gap"] = _forced_gaps(w, sel, H, biases, order, gpu)
    # make a later pick a clearly worse candidate
    taken = set(order)
    worst = [j for j in range(40) if j not in taken][-1]
    order2 = order[:-1] + [worst]
    gpu["order"][0, :len(order2)] = order2
    gpu["idx"][0, :len(order2)] = sorted(order2)
    with pytest.raises(AssertionError):
        _compare(w, sel, H, biases, gpu)
