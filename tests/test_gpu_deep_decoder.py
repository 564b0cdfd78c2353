"""GPU parity of selection with pointer decoders of several layers (layers
before the last: causal self-attention, cross-attention to the memory, GELU
FFN) against the oracle, with the selection comparison rules (bit-exact step
orders and counts except from a near-tie round on)."""
import dataclasses
import math

import numpy as np
import pytest

import _parity as PT
from paper_2609_13804_gb300 import synth as S

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_13804_gb300 import binding
    binding.lib()
    return binding


def np_(t):
    return t.cpu().numpy()


def _deep_weights(w, scale):
    """Weights with O(1) per-layer updates; the FFN matrices stay bf16 values
    (the GPU keeps them in bf16)."""
    sel = S.make_selector_weights(w, ln_affine=True)
    if scale != 1.0:
        PT.scale_decoder(sel, scale)
    for L in sel.get("lower", []):
        for n in ("Wq_s", "Wk_s", "Wv_s", "Wo_s", "Wq_c", "Wk_c", "Wv_c", "Wo_c"):
            L[n] = (L[n] / 0.02 * 0.5 / math.sqrt(L[n].shape[-1])).astype(np.float32)
        for n in ("W1", "W2"):
            L[n] = S.bf16_round((L[n] / 0.02 * 0.5 / math.sqrt(L[n].shape[-1])).astype(np.float32))
    return sel


def _deep_case(B, w, *, scale=1.0, targets=None, mean_target=None):
    sel = _deep_weights(w, scale)
    H = S.make_memory(w)
    eps_list = PT.episodes(w.n_vis, w.group_size)
    if targets is None:
        targets = S.uniform_int(w.seed, "targets", 0, w.k_max + 1, len(eps_list))
    biases = PT.calibrate_biases(H, w.n_vis, sel, k_max=w.k_max, g=1, group_size=w.group_size, targets=targets,
                                 mean_target=mean_target)
    s = w.selector
    shape = S.SelectorShape(D=s.D, D_text=s.D_text, h=s.h, n_enc_layers=0, n_dec_layers=s.n_dec_layers)
    selector = B.Selector(shape, sel, DEV)
    out = B.sp_select(selector, w.n_vis, w.n_txt, H=B.dev_f32(H, DEV), stop_bias=B.dev_f32(biases, DEV),
                      group_size=w.group_size, g=1, k_max=w.k_max)
    torch.cuda.synchronize()
    assert int(out["err"].item()) == 0
    gpu = {k: np_(out[k]) for k in ("order", "ep_count", "rounds", "margin", "gap", "idx", "count")}
    images = PT.oracle_select(H, w.n_vis, sel, k_max=w.k_max, g=1, group_size=w.group_size, biases=biases)
    replay, eps_list = PT.replayer(H, w.n_vis, sel, k_max=w.k_max, g=1, group_size=w.group_size, biases=biases)
    report = []
    near = PT.compare_selection(gpu, images, g=1, report=report, replay=replay, episodes=eps_list)
    for r in report:
        print("near-tie:", r)
    selector.close()
    return gpu, near


def _with_layers(w, n_dec):
    w.selector = dataclasses.replace(w.selector, n_dec_layers=n_dec)
    return w


@pytest.mark.parametrize("n_dec", [2, 3])
def test_deep_decoder_tiny_ragged(B, n_dec):
    w = _with_layers(S.tiny_workload(71, [37, 5, 130, 1, 64], [3, 0, 2, 1, 4], D=128, h=128, k_max=12), n_dec)
    _deep_case(B, w, scale=4.0)


def test_deep_decoder_groups_h256(B):
    w = _with_layers(S.tiny_workload(72, [300, 77, 128], [2, 2, 2], D=256, h=256, k_max=20, group_size=128), 2)
    _deep_case(B, w, scale=4.0)


def test_deep_decoder_stop_extremes(B):
    w = _with_layers(S.tiny_workload(73, [9, 20, 3], [1, 1, 1], D=128, h=128, k_max=8), 2)
    gpu, _ = _deep_case(B, w, scale=4.0, targets=[0, 8, 3])
    assert int(gpu["count"][0]) == 0
    assert int(gpu["count"][1]) == 8 and int(gpu["rounds"][1]) == 8
    assert int(gpu["count"][2]) == 3 and int(gpu["rounds"][2]) == 4


def test_deep_decoder_llava_shapes(B):
    """4 images x 576 candidates, D = 1024, h = 512, two decoder layers, cap 192."""
    w = _with_layers(S.llava15_7b_b16(), 2)
    w.n_vis, w.n_txt = w.n_vis[:4], w.n_txt[:4]
    gpu, near = _deep_case(B, w, targets=[192, 16, 64, 100])
    print("kept", gpu["count"].tolist(), "near-tie episodes", near)


def test_deep_decoder_rejects_groups_of_tokens_per_round(B):
    w = _with_layers(S.tiny_workload(74, [20], [1], D=128, h=128, k_max=8), 2)
    sel = _deep_weights(w, 4.0)
    s = w.selector
    shape = S.SelectorShape(D=s.D, D_text=s.D_text, h=s.h, n_enc_layers=0, n_dec_layers=2)
    selector = B.Selector(shape, sel, DEV)
    H = B.dev_f32(S.make_memory(w), DEV)
    with pytest.raises(B.SPError, match="UNSUPPORTED"):
        B.sp_select(selector, w.n_vis, w.n_txt, H=H, stop_bias=B.dev_f32(np.zeros(1), DEV), g=5, k_max=8)
    selector.close()
