"""Pins of the CPU oracle against things other than itself: library routines
(torch fp64 modules), closed forms, brute force and the special cases the paper's
definitions reduce to.  No GPU, no CUDA library."""
import dataclasses
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import core as O
from paper_2609_13804_gb300 import synth as S

torch.set_default_dtype(torch.float64)
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def t64(x):
    return torch.as_tensor(np.asarray(x, dtype=np.float64))


# ---------------------------------------------------------------- elementary

def test_norms_and_activations_match_torch():
    x = S.normal(1, "x", (7, 33)).astype(np.float64) * 3
    g = S.normal(1, "g", (33,)).astype(np.float64)
    b = S.normal(1, "b", (33,)).astype(np.float64)
    ref = torch.nn.functional.layer_norm(t64(x), (33,), t64(g), t64(b), 1e-5).numpy()
    np.testing.assert_allclose(O.layer_norm(x, 1e-5, g, b), ref, rtol=0, atol=1e-12)
    ref = torch.nn.functional.rms_norm(t64(x), (33,), t64(g), 1e-6).numpy()
    np.testing.assert_allclose(O.rms_norm(x, 1e-6, g), ref, rtol=0, atol=1e-12)
    np.testing.assert_allclose(O.gelu(x), torch.nn.functional.gelu(t64(x)).numpy(), atol=1e-12)
    np.testing.assert_allclose(O.silu(x), torch.nn.functional.silu(t64(x)).numpy(), atol=1e-12)


def test_gelu_closed_form_points():
    # Phi(0) = 1/2, Phi(1) = 0.8413447460685429, Phi(-1) = 0.15865525393145707
    np.testing.assert_allclose(O.gelu([0.0, 1.0, -1.0]),
                               [0.0, 0.8413447460685429, -0.15865525393145707], atol=1e-15)


@pytest.mark.parametrize("hq,hkv,causal", [(4, 4, True), (4, 2, True), (6, 1, False), (2, 2, False)])
def test_attention_matches_torch_sdpa(hq, hkv, causal):
    L, dh = 9, 8
    q = S.normal(2, "q", (L, hq * dh)).astype(np.float64)
    k = S.normal(2, "k", (L, hkv * dh)).astype(np.float64)
    v = S.normal(2, "v", (L, hkv * dh)).astype(np.float64)
    out = O.attention(q, k, v, hq, hkv, causal)
    # torch layout [heads, L, dh]; expand kv heads explicitly (group of hq/hkv queries per kv head)
    Q = t64(q).view(L, hq, dh).transpose(0, 1)
    K = t64(k).view(L, hkv, dh).transpose(0, 1).repeat_interleave(hq // hkv, dim=0)
    V = t64(v).view(L, hkv, dh).transpose(0, 1).repeat_interleave(hq // hkv, dim=0)
    ref = torch.nn.functional.scaled_dot_product_attention(Q, K, V, is_causal=causal)
    np.testing.assert_allclose(out, ref.transpose(0, 1).reshape(L, hq * dh).numpy(), atol=1e-12)


def test_attention_probability_rounding_matches_torch():
    """p_store='bf16': the softmax probabilities rounded to bf16 before they
    weight the values, as torch computes it; the rounding moves each output by
    at most 2^-8 of the largest |value| (probabilities sum to 1)."""
    L, dh, hq, hkv = 11, 8, 4, 2
    q = S.normal(6, "q", (L, hq * dh)).astype(np.float64)
    k = S.normal(6, "k", (L, hkv * dh)).astype(np.float64)
    v = S.normal(6, "v", (L, hkv * dh)).astype(np.float64)
    got = O.attention(q, k, v, hq, hkv, True, p_store="bf16")
    Q = t64(q).view(L, hq, dh).transpose(0, 1)
    K = t64(k).view(L, hkv, dh).transpose(0, 1).repeat_interleave(hq // hkv, dim=0)
    V = t64(v).view(L, hkv, dh).transpose(0, 1).repeat_interleave(hq // hkv, dim=0)
    mask = torch.triu(torch.full((L, L), float("-inf")), 1)
    P = torch.softmax(Q @ K.transpose(1, 2) / math.sqrt(dh) + mask, dim=-1)
    ref = (P.float().to(torch.bfloat16).double() @ V).transpose(0, 1).reshape(L, hq * dh).numpy()
    np.testing.assert_allclose(got, ref, atol=1e-12)
    exact = O.attention(q, k, v, hq, hkv, True)
    assert 0 < np.abs(got - exact).max() <= 2.0 ** -8 * np.abs(v).max()


def test_attention_single_token_returns_value_and_is_causal():
    dh = 4
    q = S.normal(3, "q", (5, 2 * dh)).astype(np.float64)
    k = S.normal(3, "k", (5, 2 * dh)).astype(np.float64)
    v = S.normal(3, "v", (5, 2 * dh)).astype(np.float64)
    np.testing.assert_allclose(O.attention(q[:1], k[:1], v[:1], 2, 2, True), v[:1], atol=1e-15)
    base = O.attention(q, k, v, 2, 2, True)
    k2, v2 = k.copy(), v.copy()
    k2[3:] += 5.0
    v2[3:] -= 7.0
    pert = O.attention(q, k2, v2, 2, 2, True)
    np.testing.assert_allclose(pert[:3], base[:3], atol=1e-15)
    assert np.abs(pert[3:] - base[3:]).max() > 1e-3


# ---------------------------------------------------------------- selector encoder (Eq. 3)

def test_encoder_matches_torch_transformer_encoder_layer():
    w = S.tiny_workload(4, [10], [6], D=32, D_text=48, enc_head_dim=16)
    sel = S.make_selector_weights(w, ln_affine=True)
    for L in sel["enc"]:                 # torch's bias-free layer has bias-free LayerNorms
        L["ln1_b"] = np.zeros_like(L["ln1_b"])
        L["ln2_b"] = np.zeros_like(L["ln2_b"])
    inp = S.make_inputs(w)
    X, E = inp["X"].astype(np.float64), inp["E_text"].astype(np.float64)
    s = w.selector
    Et = O.text_projection(E, sel, s.ln_eps)
    ref_Et = torch.nn.functional.layer_norm(
        torch.nn.functional.linear(t64(E), t64(sel["W_p"])), (s.D,),
        t64(sel["ln_text_g"]), t64(sel["ln_text_b"]), s.ln_eps).numpy()
    np.testing.assert_allclose(Et, ref_Et, atol=1e-12)
    H = O.encoder(X, Et, sel, s.enc_heads, s.ln_eps)

    x = t64(np.concatenate([X, Et]))[None]
    for L in sel["enc"]:
        layer = torch.nn.TransformerEncoderLayer(
            s.D, s.enc_heads, s.enc_ffn, dropout=0.0, activation="gelu", layer_norm_eps=s.ln_eps,
            batch_first=True, norm_first=True, bias=False, dtype=torch.float64)
        with torch.no_grad():
            layer.self_attn.in_proj_weight.copy_(t64(L["Wqkv"]))
            layer.self_attn.out_proj.weight.copy_(t64(L["Wo"]))
            layer.linear1.weight.copy_(t64(L["W1"]))
            layer.linear2.weight.copy_(t64(L["W2"]))
            layer.norm1.weight.copy_(t64(L["ln1_g"]))
            layer.norm2.weight.copy_(t64(L["ln2_g"]))
        layer.eval()
        with torch.no_grad():
            x = layer(x)
    np.testing.assert_allclose(H, x[0, :10].numpy(), atol=1e-10)
    assert H.shape == (10, s.D)


@pytest.mark.parametrize("store", [None, "bf16"])
def test_encoder_storage_variant_matches_torch_functional(store):
    """The encoder block assembled from torch.nn.functional (layer_norm, linear,
    sdpa over heads, gelu) in fp64, rounding to bf16 the same tensors as the
    oracle's store='bf16' (the normalised inputs, q / k / v, the attention
    output, the GELU output); residuals unrounded."""
    F = torch.nn.functional
    w = S.tiny_workload(5, [9], [4], D=32, D_text=48, enc_head_dim=8)
    sel = S.make_selector_weights(w, ln_affine=True)
    for L in sel["enc"]:
        for k in ("Wqkv", "Wo", "W1", "W2"):
            L[k] = L[k] / 0.02 * 0.2
    s = w.selector
    X = S.normal(5, "X", (9, s.D)).astype(np.float64)
    Et = S.normal(5, "Et", (4, s.D)).astype(np.float64)
    got = O.encoder(X, Et, sel, s.enc_heads, s.ln_eps, store=store)
    rnd = (lambda t: t.float().to(torch.bfloat16).double()) if store == "bf16" else (lambda t: t)
    x = t64(np.concatenate([X, Et]))
    n, D, nh = x.shape[0], s.D, s.enc_heads
    for L in sel["enc"]:
        a = rnd(F.layer_norm(x, (D,), t64(L["ln1_g"]), t64(L["ln1_b"]), s.ln_eps))
        q, k, v = rnd(F.linear(a, t64(L["Wqkv"]))).split(D, dim=1)
        heads = [t.view(n, nh, D // nh).transpose(0, 1) for t in (q, k, v)]
        o = F.scaled_dot_product_attention(*heads).transpose(0, 1).reshape(n, D)
        x = x + F.linear(rnd(o), t64(L["Wo"]))
        m = rnd(F.layer_norm(x, (D,), t64(L["ln2_g"]), t64(L["ln2_b"]), s.ln_eps))
        x = x + F.linear(rnd(F.gelu(F.linear(m, t64(L["W1"])))), t64(L["W2"]))
    np.testing.assert_allclose(got, x[:9].numpy(), rtol=0, atol=1e-10)
    if store == "bf16":
        assert np.abs(got - O.encoder(X, Et, sel, s.enc_heads, s.ln_eps)).max() > 1e-4


# ---------------------------------------------------------------- pointer decoder (Eq. 4)

def _scaled_selector(seed, N=14, D=24, h=16, scale=0.3, ln_affine=True):
    """Tiny selector whose logits are O(1) so that near-ties are rare."""
    w = S.tiny_workload(seed, [N], [3], D=D, h=h)
    sel = S.make_selector_weights(w, ln_affine=ln_affine)
    for n in ("W_in", "Wq_s", "Wk_s", "Wv_s", "Wo_s", "Wq_p", "Wk_p", "s_start", "s_stop"):
        sel[n] = (sel[n] / 0.02 * scale / math.sqrt(sel[n].shape[-1])).astype(np.float32)
    H = S.make_memory(w).astype(np.float64)
    return sel, H


def test_pointer_logits_match_torch_multihead_attention_decoder():
    """The decoder of Eq. 4 built from torch.nn.MultiheadAttention (1 head, no
    biases): causal self-attention with residual, then cross-attention to M whose
    attention probabilities are softmax(l_t + Mask_t)."""
    sel, H = _scaled_selector(5)
    N, D = H.shape
    h = sel["W_in"].shape[0]
    M = np.concatenate([H, sel["s_stop"][None].astype(np.float64)])
    hist = np.stack([sel["s_start"], M[3], M[7], M[1]]).astype(np.float64)
    ours = O.pointer_logits_from_scratch(hist, M, sel, 1e-5)

    sa = torch.nn.MultiheadAttention(h, 1, bias=False, batch_first=True)
    ca = torch.nn.MultiheadAttention(h, 1, bias=False, kdim=D, vdim=D, batch_first=True)
    with torch.no_grad():
        sa.in_proj_weight.copy_(t64(np.concatenate([sel["Wq_s"], sel["Wk_s"], sel["Wv_s"]])))
        sa.out_proj.weight.copy_(t64(sel["Wo_s"]))
        ca.q_proj_weight.copy_(t64(sel["Wq_p"]))
        ca.k_proj_weight.copy_(t64(sel["Wk_p"]))
        ca.v_proj_weight.copy_(torch.randn(h, D))
    ln1 = lambda y: torch.nn.functional.layer_norm(y, (h,), t64(sel["ln1_g"]), t64(sel["ln1_b"]), 1e-5)
    ln2 = lambda y: torch.nn.functional.layer_norm(y, (h,), t64(sel["ln2_g"]), t64(sel["ln2_b"]), 1e-5)
    with torch.no_grad():
        y = torch.nn.functional.linear(t64(hist), t64(sel["W_in"]))[None]
        causal = torch.triu(torch.full((4, 4), float("-inf")), 1)
        x = ln1(y)
        u = y + sa(x, x, x, attn_mask=causal, need_weights=False)[0]
        mask = torch.zeros(1, N + 1)
        mask[0, [3, 7, 1]] = float("-inf")
        _, p = ca(ln2(u[:, -1:]), t64(M)[None], t64(M)[None], attn_mask=mask, need_weights=True)
    logp = torch.log(p[0, 0]).numpy()
    avail = [j for j in range(N + 1) if j not in (3, 7, 1)]
    d_ours = ours[avail] - ours[avail].max()
    d_ref = logp[avail] - logp[avail].max()
    np.testing.assert_allclose(d_ours, d_ref, atol=1e-10)


def _deep_selector(seed, n_dec, N=12, D=16, h=16, scale=0.3):
    """Tiny selector with n_dec decoder layers; every decoder matrix scaled so
    that each layer moves its input by O(1)."""
    w = S.tiny_workload(seed, [N], [3], D=D, h=h)
    w.selector = dataclasses.replace(w.selector, n_dec_layers=n_dec)
    sel = S.make_selector_weights(w, ln_affine=True)
    def sc(a):
        return (a / 0.02 * scale / math.sqrt(a.shape[-1])).astype(np.float32)
    for n in ("W_in", "Wq_s", "Wk_s", "Wv_s", "Wo_s", "Wq_p", "Wk_p", "s_start", "s_stop"):
        sel[n] = sc(sel[n])
    for L in sel.get("lower", []):
        for n in ("Wq_s", "Wk_s", "Wv_s", "Wo_s", "Wq_c", "Wk_c", "Wv_c", "Wo_c", "W1", "W2"):
            L[n] = sc(L[n])
    return sel, S.make_memory(w).astype(np.float64)


@pytest.mark.parametrize("n_dec", [2, 3])
def test_deep_pointer_decoder_matches_torch_transformer_decoder_layers(n_dec):
    """Layers before the last = torch.nn.TransformerDecoderLayer (pre-norm, one
    head, no biases, GELU, FFN 4h) over the history with memory M (D = h here,
    the module's constraint); the last layer as in the one-layer pin."""
    sel, H = _deep_selector(40 + n_dec, n_dec)
    N, D = H.shape
    h = sel["W_in"].shape[0]
    M = np.concatenate([H, sel["s_stop"][None].astype(np.float64)])
    hist = np.stack([sel["s_start"], M[3], M[7], M[1], M[10]]).astype(np.float64)
    ours = O.pointer_logits_from_scratch(hist, M, sel, 1e-5)
    t = hist.shape[0]
    causal = torch.triu(torch.full((t, t), float("-inf")), 1)
    with torch.no_grad():
        y = torch.nn.functional.linear(t64(hist), t64(sel["W_in"]))[None]
        for L in sel["lower"]:
            layer = torch.nn.TransformerDecoderLayer(h, 1, dim_feedforward=4 * h, dropout=0.0, activation="gelu",
                                                     batch_first=True, norm_first=True, bias=False)
            layer.self_attn.in_proj_weight.copy_(t64(np.concatenate([L["Wq_s"], L["Wk_s"], L["Wv_s"]])))
            layer.self_attn.out_proj.weight.copy_(t64(L["Wo_s"]))
            layer.multihead_attn.in_proj_weight.copy_(t64(np.concatenate([L["Wq_c"], L["Wk_c"], L["Wv_c"]])))
            layer.multihead_attn.out_proj.weight.copy_(t64(L["Wo_c"]))
            layer.linear1.weight.copy_(t64(L["W1"]))
            layer.linear2.weight.copy_(t64(L["W2"]))
            for k in (1, 2, 3):  # bias=False drops the norms' biases too: give them back
                norm = torch.nn.LayerNorm(h, eps=1e-5)
                norm.weight.copy_(t64(L[f"ln{k}_g"]))
                norm.bias.copy_(t64(L[f"ln{k}_b"]))
                setattr(layer, f"norm{k}", norm)
            y = layer(y, t64(M)[None], tgt_mask=causal)
        sa = torch.nn.MultiheadAttention(h, 1, bias=False, batch_first=True)
        ca = torch.nn.MultiheadAttention(h, 1, bias=False, kdim=D, vdim=D, batch_first=True)
        sa.in_proj_weight.copy_(t64(np.concatenate([sel["Wq_s"], sel["Wk_s"], sel["Wv_s"]])))
        sa.out_proj.weight.copy_(t64(sel["Wo_s"]))
        # D = h: the module packs the cross-attention projections
        ca.in_proj_weight.copy_(torch.cat([t64(sel["Wq_p"]), t64(sel["Wk_p"]), torch.randn(h, D)]))
        x = torch.nn.functional.layer_norm(y, (h,), t64(sel["ln1_g"]), t64(sel["ln1_b"]), 1e-5)
        u = y + sa(x, x, x, attn_mask=causal, need_weights=False)[0]
        x2 = torch.nn.functional.layer_norm(u[:, -1:], (h,), t64(sel["ln2_g"]), t64(sel["ln2_b"]), 1e-5)
        _, p = ca(x2, t64(M)[None], t64(M)[None], need_weights=True)
    logp = torch.log(p[0, 0]).numpy()
    np.testing.assert_allclose(ours - ours.max(), logp - logp.max(), atol=1e-10)


@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("n_dec", [2, 3])
def test_deep_decoder_incremental_equals_brute_force(seed, n_dec):
    sel, H = _deep_selector(140 + seed, n_dec, N=10, D=24)
    for g in (1, 3):
        for bias in (-0.3, 0.2, -1e9):
            a = O.select_episode(H, sel, k_max=7, g=g, stop_bias=bias)
            b = O.select_episode(H, sel, k_max=7, g=g, stop_bias=bias, mode="scratch")
            assert a["order"] == b["order"] and a["stopped"] == b["stopped"]
            np.testing.assert_allclose(a["gap"], b["gap"], atol=1e-11)


@pytest.mark.parametrize("seed", range(12))
@pytest.mark.parametrize("g", [1, 3])
def test_incremental_selection_equals_brute_force(seed, g):
    sel, H = _scaled_selector(100 + seed, N=11 + seed % 5)
    N = H.shape[0]
    for bias in (-0.4, 0.0, 0.5, -1e9):
        for k_max in (3, 8, N + 3):
            a = O.select_episode(H, sel, k_max=k_max, g=g, stop_bias=bias)
            b = O.select_episode(H, sel, k_max=k_max, g=g, stop_bias=bias, mode="scratch")
            assert a["order"] == b["order"]
            assert a["stopped"] == b["stopped"]
            np.testing.assert_allclose(a["gap"], b["gap"], atol=1e-12)
            np.testing.assert_allclose(a["margin"], b["margin"], atol=1e-12)


def _exhaustive_greedy(H, sel, k_max, g, bias):
    """Brute force written from Alg. 1 without the oracle's episode loop: at every
    round rescore all N+1 candidates from scratch, then pick by a full sort."""
    N = H.shape[0]
    M = np.concatenate([H, sel["s_stop"][None].astype(np.float64)])
    hist, S_ = [sel["s_start"].astype(np.float64)], []
    while len(S_) < k_max:
        l = O.pointer_logits_from_scratch(np.stack(hist), M, sel, 1e-5)
        l[N] += bias
        cand = [(-l[j], j) for j in range(N) if j not in S_]
        if not cand:
            break
        cand.sort()
        if l[N] > -cand[0][0]:
            break
        for _, j in cand[:min(g, k_max - len(S_))]:
            S_.append(j)
            hist.append(M[j])
    return S_


@pytest.mark.parametrize("seed", range(6))
def test_selection_equals_exhaustive_greedy(seed):
    sel, H = _scaled_selector(200 + seed, N=9)
    for g in (1, 2, 5):
        for bias in (-0.3, 0.2, -1e9):
            ref = _exhaustive_greedy(H, sel, 7, g, bias)
            assert O.select_episode(H, sel, k_max=7, g=g, stop_bias=bias)["order"] == ref


def test_history_free_case_reduces_to_static_top_k():
    """With W_in = 0 every decoder token is 0, LN1 returns its bias, so queries,
    keys and values are the same at every position and the pointer query does
    not depend on the history: the policy is Eq. 1's independent top-K whose K
    is the number of static scores strictly above the STOP logit (capped)."""
    sel, H = _scaled_selector(7, N=40)
    sel["W_in"] = np.zeros_like(sel["W_in"])
    N = H.shape[0]
    h = sel["W_in"].shape[0]
    x = sel["ln1_b"].astype(np.float64)                       # LN1(0) = bias
    u = (x @ sel["Wv_s"].T.astype(np.float64)) @ sel["Wo_s"].T.astype(np.float64)
    q = O.layer_norm(u, 1e-5, sel["ln2_g"], sel["ln2_b"]) @ sel["Wq_p"].T.astype(np.float64)
    M = np.concatenate([H, sel["s_stop"][None].astype(np.float64)])
    static = (M @ sel["Wk_p"].T.astype(np.float64)) @ q / math.sqrt(h)
    order = sorted(range(N), key=lambda j: (-static[j], j))
    for bias in (-0.5, 0.0, 0.3, -1e9):
        stop = static[N] + bias
        K = sum(1 for j in range(N) if static[j] > stop)
        for k_max in (5, 12, 50):
            for g in (1, 5):
                # Sec. 3.5: STOP is only checked at the start of a round, so with
                # g tokens per round the kept set is the top g*ceil(K/g) (capped)
                want = order[:min(g * math.ceil(K / g), N, k_max)]
                r = O.select_episode(H, sel, k_max=k_max, g=g, stop_bias=bias)
                assert r["order"] == want
                k = len(want)
                stopped = k < k_max
                assert r["rounds"] == math.ceil(k / g) + (1 if stopped else 0)


@pytest.mark.parametrize("seed", range(8))
def test_selection_invariants_and_bias_monotonicity(seed):
    sel, H = _scaled_selector(300 + seed, N=30)
    N = H.shape[0]
    base = O.select_episode(H, sel, k_max=N, g=1, stop_bias=-1e9)
    gaps = np.array(base["gap"])
    prev_k = None
    for bias in np.linspace(-1.5, 1.5, 13):
        r = O.select_episode(H, sel, k_max=20, g=1, stop_bias=bias)
        o = r["order"]
        assert len(set(o)) == len(o) and r["count"] == len(o) <= 20
        assert all(0 <= i < N for i in o)
        # the trajectory does not depend on the bias until STOP wins
        assert o == base["order"][:len(o)]
        # closed form: K(b) = first round t with gap_t < b, minus one; capped by k_max
        t = next((i for i, gp in enumerate(gaps) if gp < bias), len(gaps))
        assert r["count"] == min(t, 20)
        if prev_k is not None:
            assert r["count"] <= prev_k
        prev_k = r["count"]
    assert list(O.restore(o)) == sorted(o)


def test_selection_extremes():
    sel, H = _scaled_selector(9, N=6)
    assert O.select_episode(H, sel, k_max=4, stop_bias=1e9)["count"] == 0
    r = O.select_episode(H, sel, k_max=100, stop_bias=-1e9)
    assert sorted(r["order"]) == list(range(6)) and r["stopped"]
    r = O.select_episode(H[:1], sel, k_max=3, stop_bias=-1e9)
    assert r["order"] == [0] and r["rounds"] == 2
    r = O.select_episode(H, sel, k_max=5, g=50, stop_bias=-1e9)
    assert r["count"] == 5 and r["rounds"] == 1
    img = O.select_image(H, sel, k_max=2, g=1, group_size=1, stop_bias=[-1e9] * 6)
    assert list(img["idx"]) == list(range(6))


def test_candidate_groups_are_independent_episodes():
    sel, H = _scaled_selector(10, N=23)
    biases = [-0.1, 0.2, -1e9]
    img = O.select_image(H, sel, k_max=4, g=2, group_size=10, stop_bias=biases)
    want = []
    for e, s in enumerate((0, 10, 20)):
        r = O.select_episode(H[s:s + 10], sel, k_max=4, g=2, stop_bias=biases[e])
        want += [s + i for i in r["order"]]
    assert list(img["idx"]) == sorted(want)


@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("g", [1, 3])
def test_forcing_the_own_order_changes_nothing(seed, g):
    sel, H = _scaled_selector(400 + seed, N=17)
    for bias in (-0.3, 0.1, -1e9):
        for k_max in (5, 40):
            r = O.select_episode(H, sel, k_max=k_max, g=g, stop_bias=bias)
            f = O.select_episode(H, sel, k_max=k_max, g=g, stop_bias=bias, force=r["order"])
            assert f["order"] == r["order"] and f["rounds"] == r["rounds"] and f["stopped"] == r["stopped"]
            assert f["gap"] == r["gap"] and f["margin"] == r["margin"]
            assert all(x == 0.0 for x in f["slack"])


@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("g", [1, 2])
def test_forced_slack_equals_brute_force_rescoring(seed, g):
    """Along an arbitrary forced trajectory the slack of every round is the
    distance of the forced decision from an optimal one, rescoring all
    candidates from scratch over the forced history (written from Alg. 1 and
    Eq. 11, without the oracle's episode loop)."""
    sel, H = _scaled_selector(500 + seed, N=12)
    N = H.shape[0]
    rng = np.random.default_rng(seed)
    k_max, bias = 9, -0.2
    force = [int(x) for x in rng.permutation(N)[:int(rng.integers(0, k_max + 1))]]
    f = O.select_episode(H, sel, k_max=k_max, g=g, stop_bias=bias, force=force)
    M = np.concatenate([H, sel["s_stop"][None].astype(np.float64)])
    hist, done, want = [sel["s_start"].astype(np.float64)], [], []
    while len(done) < k_max:
        l = O.pointer_logits_from_scratch(np.stack(hist), M, sel, 1e-5)
        l[N] += bias
        av = sorted((l[j] for j in range(N) if j not in done), reverse=True)
        if not av:
            want.append(0.0)
            break
        if len(done) == len(force):
            want.append(max(0.0, av[0] - l[N]))
            break
        take = min(g, k_max - len(done), len(av))
        U = force[len(done):len(done) + take]
        lu = [l[u] for u in U]
        rise = max([lu[i + 1] - lu[i] for i in range(take - 1)] + [0.0])
        want.append(max(0.0, av[take - 1] - min(lu), l[N] - av[0], rise))
        done += U
        hist += [M[u] for u in U]
    assert f["order"] == force
    np.testing.assert_allclose(f["slack"], want, atol=1e-12)
    assert max(want) > 0.0  # a random trajectory is not the greedy one
    with pytest.raises(ValueError):
        O.select_episode(H, sel, k_max=k_max, g=1, stop_bias=bias, force=[0, 0])


# ---------------------------------------------------------------- compaction (Alg. 1 step 5)

def test_compaction_golden_fixture():
    with open(os.path.join(GOLDEN, "compact_tiny.json")) as f:
        gold = json.load(f)
    packed, cu, pos = O.compact(np.array(gold["X"]), gold["n_vis"], gold["idx"],
                                np.array(gold["text"]), gold["n_txt"])
    np.testing.assert_array_equal(packed, np.array(gold["packed"]))
    np.testing.assert_array_equal(cu, gold["cu_seqlens"])
    np.testing.assert_array_equal(pos, gold["pos"])


# ---------------------------------------------------------------- RoPE and the LM layer

def test_rope_is_a_rotation_with_relative_positions():
    dh, H = 8, 2
    x = S.normal(11, "x", (5, H * dh)).astype(np.float64)
    pos = np.array([0, 1, 2, 7, 100])
    r = O.rope(x, pos, H, dh, 1e4)
    np.testing.assert_allclose(r[0], x[0], atol=1e-15)
    xr, rr = x.reshape(5, H, dh), r.reshape(5, H, dh)
    for i in range(dh // 2):   # each (i, i + dh/2) pair keeps its length
        np.testing.assert_allclose(xr[..., i] ** 2 + xr[..., i + 4] ** 2,
                                   rr[..., i] ** 2 + rr[..., i + 4] ** 2, atol=1e-12)
    # pair 0 rotates by exactly pos radians (inv_freq_0 = 1)
    e = np.zeros((1, dh)); e[0, 0] = 1.0
    rot = O.rope(e, np.array([1.0]), 1, dh, 1e4)
    np.testing.assert_allclose([rot[0, 0], rot[0, 4]], [math.cos(1.0), math.sin(1.0)], atol=1e-15)
    # <R_m q, R_n k> depends only on m - n
    q = S.normal(11, "q", (1, dh)).astype(np.float64)
    k = S.normal(11, "k", (1, dh)).astype(np.float64)
    d1 = O.rope(q, [5], 1, dh, 1e4) @ O.rope(k, [2], 1, dh, 1e4).T
    d2 = O.rope(q, [33], 1, dh, 1e4) @ O.rope(k, [30], 1, dh, 1e4).T
    np.testing.assert_allclose(d1, d2, atol=1e-12)


def test_mrope_reduces_to_rope_and_keeps_componentwise_relative_positions():
    dh, H, sec = 16, 2, (2, 3, 3)
    x = S.normal(12, "x", (6, H * dh)).astype(np.float64)
    p1 = np.array([0, 1, 2, 7, 100, 3])
    # equal components: the 1-D rotation
    np.testing.assert_allclose(O.mrope(x, np.repeat(p1[:, None], 3, 1), H, dh, 1e4, sec),
                               O.rope(x, p1, H, dh, 1e4), atol=1e-13)
    # one section holding every pair: the 1-D rotation by that component
    p3 = np.stack([p1, 5 * p1 + 1, 3 - p1], axis=1)
    for c in range(3):
        one = [0, 0, 0]
        one[c] = dh // 2
        np.testing.assert_allclose(O.mrope(x, p3, H, dh, 1e4, one), O.rope(x, p3[:, c], H, dh, 1e4), atol=1e-13)
    # pair lengths are kept
    r = O.mrope(x, p3, H, dh, 1e4, sec).reshape(6, H, dh)
    xr = x.reshape(6, H, dh)
    np.testing.assert_allclose(xr[..., :8] ** 2 + xr[..., 8:] ** 2, r[..., :8] ** 2 + r[..., 8:] ** 2, atol=1e-12)
    # <R(a) q, R(b) k> depends only on a - b, component by component
    q = S.normal(12, "q", (1, dh)).astype(np.float64)
    k = S.normal(12, "k", (1, dh)).astype(np.float64)
    a, b, sh = np.array([[2, 5, 9]]), np.array([[0, 1, 4]]), np.array([[11, -3, 40]])
    d1 = O.mrope(q, a, 1, dh, 1e4, sec) @ O.mrope(k, b, 1, dh, 1e4, sec).T
    d2 = O.mrope(q, a + sh, 1, dh, 1e4, sec) @ O.mrope(k, b + sh, 1, dh, 1e4, sec).T
    np.testing.assert_allclose(d1, d2, atol=1e-12)


def _full_sequence_positions(n_vis, grid_w, n_txt):
    """The unpruned sequence's (t, h, w) rows, by walking the grid row by row."""
    rows, top = [], 0
    for i in range(n_vis):
        r, c = i // grid_w, i % grid_w
        rows.append((0, r, c))
        top = max(top, r, c)
    for j in range(n_txt):
        rows.append((top + 1 + j,) * 3)
    return np.array(rows, dtype=np.float64)


@pytest.mark.parametrize("n,gw,nt", [(16, 4, 3), (12, 4, 5), (10, 4, 2), (576, 24, 7), (7, 7, 1)])
def test_mrope_positions_are_the_full_sequence_rows(n, gw, nt):
    full = _full_sequence_positions(n, gw, nt)
    np.testing.assert_array_equal(O.mrope_positions(np.arange(n), n, gw, nt), full)
    kept = np.sort(np.random.default_rng(n).choice(n, size=max(1, n // 3), replace=False))
    got = O.mrope_positions(kept, n, gw, nt)
    np.testing.assert_array_equal(got, np.concatenate([full[kept], full[n:]]))
    assert O.mrope_positions([], n, gw, nt).shape == (nt, 3)


def test_decode_with_rotary_positions_equals_mrope_prefill():
    """A generated text token (equal components) at position p after an mRoPE
    prefix: decode_step with rope_pos = p is the prefill over the extended
    sequence with that row's 3-D position (p, p, p)."""
    w = S.tiny_workload(13, [6, 4], [2, 3], d=32, n_heads=4, n_kv_heads=2, head_dim=16, ffn=40)
    m = dataclasses.replace(w.model, mrope_section=(2, 3, 3))
    layers = [S.make_layer_weights(w, l, norm_affine=True) for l in range(2)]
    for L in layers:
        for k in ("Wqkv", "Wo", "Wgu", "Wdown"):
            L[k] = L[k] / 0.02 * 0.15
    lens, grids = [8, 7], [3, 2]
    kept = [[0, 2, 3, 5, 6, 7], [0, 1, 3, 4]]
    n_img = [8, 5]
    pos3 = [O.mrope_positions(k, n, gw, t) for k, n, gw, t in zip(kept, n_img, grids, [2, 3])]
    x = S.normal(13, "x", (sum(lens), 32)).astype(np.float64)
    cu = np.array([0, 8, 15])
    kv = []
    O.prefill(x, layers, m, cu, np.concatenate(pos3), kv_out=kv)
    cache = O.cache_from_prefill(kv, cu)
    xn = S.normal(13, "xn", (2, 32)).astype(np.float64)
    nxt = [int(p[-1, 0]) + 1 for p in pos3]
    hid, _ = O.decode_step(xn, layers, m, cache, rope_pos=nxt)
    for b in range(2):
        xs = np.concatenate([x[cu[b]:cu[b + 1]], xn[b:b + 1]])
        ps = np.concatenate([pos3[b], [[nxt[b]] * 3]])
        ref = O.prefill(xs, layers, m, [0, len(xs)], ps)
        np.testing.assert_allclose(hid[b], ref[-1], atol=1e-10)


def _tiny_lm(seed, hq=4, hkv=2):
    w = S.tiny_workload(seed, [5, 3], [2, 4], d=32, n_heads=hq, n_kv_heads=hkv, head_dim=8, ffn=40)
    L = S.make_layer_weights(w, 0, norm_affine=True)
    for k in ("Wqkv", "Wo", "Wgu", "Wdown"):
        L[k] = L[k] / 0.02 * 0.15
    return w, L


def test_prefill_layer_zero_output_weights_is_identity():
    w, L = _tiny_lm(12)
    L["Wo"] = np.zeros_like(L["Wo"])
    L["Wdown"] = np.zeros_like(L["Wdown"])
    x = S.normal(12, "x", (14, 32)).astype(np.float64)
    cu, pos = [0, 7, 14], np.r_[np.arange(7), np.arange(7)]
    np.testing.assert_allclose(O.prefill_layer(x, L, w.model, cu, pos), x, atol=1e-15)


def test_prefill_layer_uniform_attention_closed_form():
    """Wq = 0 makes every causal score equal: the attention output at position p
    is the mean of the values at 0..p of its own sequence."""
    w, L = _tiny_lm(13, hq=4, hkv=4)
    m = w.model
    dq = m.n_heads * m.head_dim
    L["Wqkv"][:dq] = 0.0
    L["Wo"] = np.eye(m.d, dq)
    L["Wdown"] = np.zeros_like(L["Wdown"])
    x = S.normal(13, "x", (9, m.d)).astype(np.float64)
    cu, pos = [0, 4, 9], np.r_[np.arange(4), np.arange(5)]
    out = O.prefill_layer(x, L, m, cu, pos)
    v = O.rms_norm(x, m.rms_eps, L["attn_norm"]) @ L["Wqkv"][2 * dq:].astype(np.float64).T
    want = np.zeros_like(v)
    for s, e in ((0, 4), (4, 9)):
        for p in range(s, e):
            want[p] = v[s:p + 1].mean(axis=0)
    np.testing.assert_allclose(out - x, want, atol=1e-12)


def _torch_llama_layer(h, L, m, lens, store=None):
    """A Llama decoder layer over packed sequences assembled from
    torch.nn.functional in fp64: rms_norm, linear, rotary as a complex rotation
    of the (i, i + dh/2) pairs (torch.polar), scaled_dot_product_attention with
    the key / value heads repeated for their query groups, silu.  With
    store='bf16' the same tensors the oracle stores as bf16 are rounded."""
    F = torch.nn.functional
    rnd = (lambda t: t.float().to(torch.bfloat16).double()) if store == "bf16" else (lambda t: t)
    dq, dkv, half = m.n_heads * m.head_dim, m.n_kv_heads * m.head_dim, m.head_dim // 2
    Wq, Wk, Wv = t64(L["Wqkv"]).split([dq, dkv, dkv])
    Wg, Wu = t64(L["Wgu"]).split([m.ffn, m.ffn])
    inv = m.rope_theta ** (-2.0 * torch.arange(half, dtype=torch.float64) / m.head_dim)
    H, out, s0 = t64(h), [], 0
    for n in lens:
        hs = H[s0:s0 + n]
        s0 += n
        rot = torch.polar(torch.ones(n, half), torch.arange(n, dtype=torch.float64)[:, None] * inv[None, :])

        def rope(t):
            z = torch.complex(t[..., :half], t[..., half:]) * rot[:, None, :]
            return torch.cat([z.real, z.imag], dim=-1)

        x = rnd(F.rms_norm(hs, (m.d,), t64(L["attn_norm"]), m.rms_eps))
        q = rnd(rope(F.linear(x, Wq).view(n, m.n_heads, m.head_dim)))
        k = rnd(rope(F.linear(x, Wk).view(n, m.n_kv_heads, m.head_dim)))
        v = rnd(F.linear(x, Wv).view(n, m.n_kv_heads, m.head_dim))
        rep = m.n_heads // m.n_kv_heads
        o = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1).repeat_interleave(rep, 0),
                                           v.transpose(0, 1).repeat_interleave(rep, 0), is_causal=True)
        hs = hs + F.linear(rnd(o.transpose(0, 1).reshape(n, dq)), t64(L["Wo"]))
        x2 = rnd(F.rms_norm(hs, (m.d,), t64(L["mlp_norm"]), m.rms_eps))
        hs = hs + F.linear(rnd(F.silu(F.linear(x2, Wg)) * F.linear(x2, Wu)), t64(L["Wdown"]))
        out.append(hs)
    return torch.cat(out).numpy()


@pytest.mark.parametrize("hq,hkv,store", [(4, 2, None), (4, 4, None), (6, 1, None), (4, 2, "bf16")])
def test_prefill_layer_matches_torch_llama_layer(hq, hkv, store):
    """The whole LM layer, attention and SwiGLU halves with their residuals,
    against the torch composition: GQA, ragged sequences (one of length 1),
    non-trivial norm gains, weights large enough that the MLP moves the
    residual as much as the attention does."""
    w = S.tiny_workload(19, [5], [2], d=48, n_heads=hq, n_kv_heads=hkv, head_dim=8, ffn=56)
    m = w.model
    L = S.make_layer_weights(w, 0, norm_affine=True)
    for k in ("Wqkv", "Wo", "Wgu", "Wdown"):
        L[k] = L[k] / 0.02 * 0.2
    lens = [5, 1, 9, 4]
    x = S.normal(19, "x", (sum(lens), m.d)).astype(np.float64)
    cu = np.r_[0, np.cumsum(lens)]
    pos = np.concatenate([np.arange(n) for n in lens])
    got = O.prefill_layer(x, L, m, cu, pos, store=store)
    want = _torch_llama_layer(x, L, m, lens, store=store)
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-10)
    # both halves move the residual: the pin sees the MLP, not only the attention
    L0 = dict(L, Wdown=np.zeros_like(L["Wdown"]))
    assert np.abs(O.prefill_layer(x, L0, m, cu, pos) - got).max() > 0.1


@pytest.mark.parametrize("store,mrope", [(None, False), ("bf16", False), (None, True)])
def test_prefill_layer_rows_equals_the_whole_layer(store, mrope):
    """The row-sampled layer (keys / values of the whole sequence, the rest at
    the chosen rows) equals the whole layer at those rows."""
    w = S.tiny_workload(20, [5], [2], d=32, n_heads=4, n_kv_heads=2, head_dim=8, ffn=40)
    m = w.model
    if mrope:
        m = dataclasses.replace(m, mrope_section=(2, 1, 1))
    L = S.make_layer_weights(w, 0, norm_affine=True)
    for k in ("Wqkv", "Wo", "Wgu", "Wdown"):
        L[k] = L[k] / 0.02 * 0.2
    lens = [7, 1, 12, 5]
    T = sum(lens)
    x = S.normal(20, "x", (T, m.d)).astype(np.float64)
    cu = np.r_[0, np.cumsum(lens)]
    pos = np.concatenate([np.arange(n) for n in lens])
    if mrope:
        pos = np.stack([pos, pos // 3, pos % 3], axis=1).astype(np.float64)
    full = O.prefill_layer(x, L, m, cu, pos, store=store)
    rows = np.array([0, 3, 6, 7, 8, 9, 15, 19, 20, 24])
    got = O.prefill_layer_rows(x, L, m, cu, pos, rows, store=store)
    np.testing.assert_allclose(got, full[rows], rtol=0, atol=1e-10 if store is None else 1e-2)
    if store == "bf16":  # a rounding boundary may flip between the two matmul shapes, rarely
        assert np.mean(np.abs(got - full[rows]) < 1e-10) > 0.95


def test_prefill_varlen_isolation_and_causality():
    w, L = _tiny_lm(14)
    m = w.model
    x = S.normal(14, "x", (11, m.d)).astype(np.float64)
    cu, pos = [0, 6, 11], np.r_[np.arange(6), np.arange(5)]
    both = O.prefill(x, [L, L], m, cu, pos)
    alone0 = O.prefill(x[:6], [L, L], m, [0, 6], np.arange(6))
    alone1 = O.prefill(x[6:], [L, L], m, [0, 5], np.arange(5))
    np.testing.assert_allclose(both, np.concatenate([alone0, alone1]), atol=1e-12)
    x2 = x.copy()
    x2[3:6] += 1.0
    pert = O.prefill(x2, [L, L], m, cu, pos)
    np.testing.assert_allclose(pert[:3], both[:3], atol=1e-12)
    np.testing.assert_allclose(pert[6:], both[6:], atol=1e-12)


def test_prefill_fp32_accumulation_variant_is_fp32_close():
    """acc='fp32' only lowers the projections' precision: without storage
    rounding it matches the fp64 layer to fp32 round-off, and it is not the
    fp64 layer bit for bit (the option reaches the matmuls)."""
    w, L = _tiny_lm(16)
    m = w.model
    x = S.normal(16, "x", (10, m.d)).astype(np.float64)
    cu, pos = [0, 10], np.arange(10)
    a = O.prefill(x, [L, L], m, cu, pos)
    b = O.prefill(x, [L, L], m, cu, pos, acc="fp32")
    np.testing.assert_allclose(b, a, rtol=1e-4, atol=1e-5)
    assert np.abs(b - a).max() > 0.0


@pytest.mark.parametrize("store", [None, "bf16"])
def test_decode_step_equals_prefill_over_the_extended_sequences(store):
    """A generation step over the prefill's cache gives, for every sequence, the
    hidden state the prefill itself computes at that position when the new
    token is appended to the packed sequence (and the cache grows by exactly
    that position's keys / values)."""
    w, L = _tiny_lm(17, hq=4, hkv=2)
    m = w.model
    layers = [L, _tiny_lm(18, hq=4, hkv=2)[1]]
    lens = [5, 1, 9]
    x = S.normal(17, "x", (sum(lens), m.d)).astype(np.float64)
    x_new = S.normal(17, "x_new", (len(lens), m.d)).astype(np.float64)
    cu = np.r_[0, np.cumsum(lens)]
    pos = np.concatenate([np.arange(n) for n in lens])
    kv = []
    O.prefill(x, layers, m, cu, pos, store=store, kv_out=kv)
    cache = O.cache_from_prefill(kv, cu)
    got, grown = O.decode_step(x_new, layers, m, cache, store=store)
    # the same tokens as one longer prefill
    ext = np.concatenate([np.concatenate([x[cu[b]:cu[b + 1]], x_new[b:b + 1]]) for b in range(len(lens))])
    cu2 = np.r_[0, np.cumsum([n + 1 for n in lens])]
    pos2 = np.concatenate([np.arange(n + 1) for n in lens])
    kv2 = []
    full = O.prefill(ext, layers, m, cu2, pos2, store=store, kv_out=kv2)
    np.testing.assert_allclose(got, full[cu2[1:] - 1], rtol=0, atol=1e-10)
    for l in range(len(layers)):
        for b in range(len(lens)):
            np.testing.assert_allclose(grown[l][b][0], kv2[l][0][cu2[b]:cu2[b + 1]], atol=1e-12)
            np.testing.assert_allclose(grown[l][b][1], kv2[l][1][cu2[b]:cu2[b + 1]], atol=1e-12)


def test_projector_forms():
    w = S.tiny_workload(15, [4], [2], D=12, d=20)
    head = S.make_model_head(w)
    x = S.normal(15, "x", (3, 12)).astype(np.float64)
    W1, W2 = head["proj_W1"].astype(np.float64), head["proj_W2"].astype(np.float64)
    ref = torch.nn.Sequential(torch.nn.Linear(12, 20, bias=False), torch.nn.GELU(),
                              torch.nn.Linear(20, 20, bias=False))
    with torch.no_grad():
        ref[0].weight.copy_(t64(W1))
        ref[2].weight.copy_(t64(W2))
        want = ref(t64(x)).numpy()
    np.testing.assert_allclose(O.projector(x, head), want, atol=1e-12)


def test_bf16_storage_rounding_matches_torch():
    x = np.concatenate([S.normal(16, "x", (4000,)) * 10 ** k for k in range(-6, 6)]).astype(np.float64)
    x = np.concatenate([x, [0.0, -0.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, 65504.0, 1e-40]])
    ref = torch.tensor(x, dtype=torch.float64).to(torch.float32).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(O.round_bf16(x), ref)
    # storage rounding only moves values by at most half a bf16 ulp
    w, L = _tiny_lm(17)
    xin = S.normal(17, "x", (9, 32)).astype(np.float64)
    cu, pos = [0, 9], np.arange(9)
    a = O.prefill_layer(xin, L, w.model, cu, pos)
    b = O.prefill_layer(xin, L, w.model, cu, pos, store="bf16")
    assert 0 < np.abs(a - b).max() < 0.05 * np.abs(a).max()
