"""GPU parity at the sequence lengths the workloads run: one decoder layer over
packed sequences of 624 to 4,160 tokens (the full 16-image prefix of the
LLaVA-1.5-7B batch, the AnyRes pruned and full lengths, the Qwen2.5-VL / InternVL
GQA lengths) and the cross-modal encoder at the 3,584-wide selector.

The GPU runs the whole layer over every packed row; the oracle, for which a
layer over thousands of rows is too slow, computes sampled rows one by one
(prefill_layer_rows: keys and values of the whole sequence, everything else at
the chosen rows): both sides of every 128-row tile boundary, the first and last
rows of each sequence, and seeded random rows.  Tolerance: max-abs 3e-2 and
mean-rel 1e-2 against the oracle with bf16 storage of the activations, mean-rel
1e-2 against the pure fp64 oracle (max-abs printed).  The encoder memory (fp32
rows) is held to max-abs / RMS 1e-2 against the oracle with bf16 storage and
mean-rel 1e-2 against the pure fp64 oracle."""
import numpy as np
import pytest

import _parity as PT
from oracle import core as O
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
    if t.dtype == torch.bfloat16:
        return t.float().cpu().numpy()
    return t.cpu().numpy()


def sample_rows(lens, seed, n_random=12):
    """Packed indices of the sampled rows of every sequence."""
    rng = np.random.default_rng(seed)
    out, s0 = [], 0
    for n in lens:
        pick = {0, 1, n - 2, n - 1}
        for t in range(128, n, 128):
            pick |= {t - 1, t}
        pick |= {int(x) for x in rng.integers(0, n, n_random)}
        out += [s0 + p for p in sorted(pick) if 0 <= p < n]
        s0 += n
    return np.array(out, dtype=np.int64)


def _layer_case(B, w, lens, name):
    m = w.model
    L = S.make_layer_weights(w, 0, norm_affine=True)
    head = S.make_model_head(w, norm_affine=True)
    model = B.Model(m, [L], head, DEV, max_pos=max(lens) + 8)
    T = int(sum(lens))
    x = S.bf16_round(S.normal(w.seed, name, (T, m.d), 0.5))
    cu, pos = PT.lens_cu_pos(lens)
    out = B.sp_prefill(model, x=B.dev_bf16(x, DEV), cu_seqlens=torch.from_numpy(cu.astype(np.int32)).to(DEV),
                       pos=torch.from_numpy(pos.astype(np.int32)).to(DEV), B=len(lens), T_cap=T,
                       max_seqlen_cap=max(lens))
    torch.cuda.synchronize()
    assert int(out["err"].item()) == 0
    got = np_(out["hidden"])[:T]
    model.close()
    assert np.all(np.isfinite(got))
    rows = sample_rows(lens, w.seed)
    g = got[rows]
    ref = O.final_norm(O.prefill_layer_rows(x, L, m, cu, pos, rows, store="bf16"), m, head["final_norm"])
    r = PT.hidden_close(g, ref, f"{w.name} {name}")
    ref64 = O.final_norm(O.prefill_layer_rows(x, L, m, cu, pos, rows), m, head["final_norm"])
    r64 = PT.mean_rel_only(g, ref64, f"{w.name} {name}")
    print(f"{w.name} one layer, lengths {lens}, {len(rows)} sampled rows: vs bf16-storage oracle max-abs %.3e "
          "mean-rel %.3e | vs fp64 oracle max-abs %.3e mean-rel %.3e" % (r + r64))


def test_prefill_full_prefix_16x624_llama7b_dims(B):
    """The headline's full-prefix comparison: 16 sequences of 576 + 48 tokens."""
    _layer_case(B, S.llava15_7b_b16(), [624] * 16, "full624")


def test_prefill_anyres_lengths_llama7b_dims(B):
    """AnyRes pruned lengths (kept 80..640 + 64 text) and one full 2,944-token
    sequence (5 tiles x 576 + 64)."""
    _layer_case(B, S.llavanext_anyres_b8(), [144, 384, 704, 521, 2944], "anyres")


def test_prefill_long_gqa_qwen_dims(B):
    """GQA 28/4 at d = 3584, theta 1e6: 2,304-, 3,424- and 4,160-token sequences."""
    _layer_case(B, S.qwen25vl_varres_b8(), [2304, 3424, 4160], "gqa_long")


def test_encoder_memory_qwen_dims(B):
    """The 2-block cross-modal encoder at D = 3584 (56 heads of 64, FFN 14,336)
    over one 1,024-candidate image and its 64 text tokens, non-causal."""
    w = S.qwen25vl_varres_b8()
    w.n_vis, w.n_txt = [1024], [64]
    s = w.selector
    sel = S.make_selector_weights(w, ln_affine=True)
    inp = S.make_inputs(w)
    selector = B.Selector(s, sel, DEV)
    out = B.sp_select(selector, w.n_vis, w.n_txt, X=B.dev_bf16(inp["X"], DEV), E_text=B.dev_bf16(inp["E_text"], DEV),
                      stop_bias=B.dev_f32(np.zeros(1), DEV), group_size=0, g=1, k_max=4, memory=True)
    torch.cuda.synchronize()
    assert int(out["err"].item()) == 0
    got = np_(out["memory"])
    selector.close()
    Et = O.text_projection(inp["E_text"], sel, s.ln_eps, s.g_text)
    ref = O.encoder(inp["X"], Et, sel, s.D // s.enc_head_dim, s.ln_eps, store="bf16")
    rel = np.abs(got - ref).max() / np.sqrt((ref ** 2).mean())
    ref64 = O.encoder(inp["X"], Et, sel, s.D // s.enc_head_dim, s.ln_eps)
    d64 = np.abs(got - ref64)
    rel64, mrel64 = d64.max() / np.sqrt((ref64 ** 2).mean()), d64.mean() / np.abs(ref64).mean()
    print(f"encoder D=3584, 1024 + 64 rows: vs bf16-storage oracle max-abs / rms {rel:.3e} | vs fp64 oracle "
          f"max-abs / rms {rel64:.3e} mean-rel {mrel64:.3e}")
    assert rel <= PT.HID_MAX_ABS, rel
    assert mrel64 <= PT.HID_MEAN_REL, mrel64


def test_pipeline_equals_its_stages_qwen_dims(B):
    """The chained call at the Qwen2.5-VL-7B dims (8 images of 256..4,096
    tokens; the 3,584-wide two-block encoder, whose 56 heads of 64 over up to
    4,160 rows take the streamed attention kernel; groups of 1,024 with g = 5;
    GQA 28/4; no projector), one decoder layer: the same bytes as its stages
    called one by one (sp_select -> sp_compact -> sp_prefill).  Weights and
    inputs are drawn on the device (both sides read the same bytes); STOP biases
    keep about 11% of every group."""
    import dataclasses
    import os
    import sys
    sys.path.insert(0, os.path.abspath(os.path.join(os.path.dirname(__file__), "..")))
    import bench
    w = S.qwen25vl_varres_b8()
    w = dataclasses.replace(w, model=dataclasses.replace(w.model, n_layers=1))
    s = w.selector
    gen = torch.Generator(device=DEV)
    gen.manual_seed(2604)
    sel = B.Selector(s, bench.device_selector_weights(s, DEV, gen, torch), DEV)
    model = bench.device_model(B, w.model, DEV, gen, torch, max_pos=4096 + 256)
    X = torch.randn((sum(w.n_vis), s.D), device=DEV, generator=gen).to(torch.bfloat16)
    E = (torch.randn((sum(w.n_txt), s.D_text), device=DEV, generator=gen) * 0.02).to(torch.bfloat16)
    eps = w.episodes()
    cal = B.sp_select(sel, w.n_vis, w.n_txt, X=X, E_text=E, stop_bias=B.dev_f32(np.full(len(eps), -1e30), DEV),
                      group_size=w.group_size, g=w.g, k_max=w.k_max)
    torch.cuda.synchronize()
    gaps, rounds = np_(cal["gap"]), np_(cal["rounds"])
    targets, _ = bench.episode_targets(w)
    biases, _ = S.stop_biases([gaps[e, :rounds[e]] for e in range(len(eps))], targets, g=w.g, k_max=w.k_max,
                              n_cand=[n for (_, _, n) in eps])
    bd = B.dev_f32(biases, DEV)
    pipe = B.Pipeline(sel, model, w.n_vis, w.n_txt, group_size=w.group_size, g=w.g, k_max=w.k_max)
    pipe(X, E, bd)
    r = B.sp_select(sel, w.n_vis, w.n_txt, X=X, E_text=E, stop_bias=bd, group_size=w.group_size, g=w.g,
                    k_max=w.k_max, k_cap=pipe.k_cap, traces=False)
    c = B.sp_compact(w.n_vis, w.n_txt, X=X, text=E, idx=r["idx"], count=r["count"], k_cap=pipe.k_cap)
    max_len = max(min(n, pipe.k_cap) + t for n, t in zip(w.n_vis, w.n_txt))
    p = B.sp_prefill(model, x=c["packed"], cu_seqlens=c["cu_seqlens"], pos=c["pos"], B=w.B, T_cap=c["T_cap"],
                     max_seqlen_cap=max_len)
    torch.cuda.synchronize()
    assert int(pipe.err.item()) == 0 and int(c["err"].item()) == 0 and int(p["err"].item()) == 0
    counts = np_(pipe.count)
    assert counts.tolist() == np_(r["count"]).tolist()
    assert 0.05 * sum(w.n_vis) < counts.sum() < 0.2 * sum(w.n_vis)
    np.testing.assert_array_equal(np_(pipe.idx), np_(r["idx"]))
    cu = np_(pipe.cu)
    np.testing.assert_array_equal(cu, np_(c["cu_seqlens"]))
    T = int(cu[-1])
    h = np_(pipe.hidden)[:T]
    assert np.isfinite(h).all()
    np.testing.assert_array_equal(h, np_(p["hidden"])[:T])
    print("qwen-dims pipeline: kept", counts.tolist(), "of", w.n_vis)
    sel.close()
    model.close()
