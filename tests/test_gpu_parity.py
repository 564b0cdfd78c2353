"""GPU parity: every stage of the path through the C ABI against the CPU oracle
on the same seeded inputs (stage-local: each stage is fed seeded inputs, never
another stage's GPU output)."""
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


# ------------------------------------------------------------------ selection (Eq. 4, Eq. 11, Alg. 1)

def _run_select_case(B, w, *, scale=1.0, ln_affine=True, targets=None, seed_bias=0, mean_target=None):
    s = w.selector
    sel = S.make_selector_weights(w, ln_affine=ln_affine)
    if scale != 1.0:
        PT.scale_decoder(sel, scale)
    H = S.make_memory(w)
    eps_list = PT.episodes(w.n_vis, w.group_size)
    if targets is None:
        t = S.uniform_int(w.seed + seed_bias, "targets", 0, w.k_max + 1, len(eps_list))
    else:
        t = targets
    biases = PT.calibrate_biases(H, w.n_vis, sel, k_max=w.k_max, g=w.g, group_size=w.group_size, targets=t,
                                 mean_target=mean_target)
    shape = S.SelectorShape(D=s.D, D_text=s.D_text, h=s.h, n_enc_layers=0)
    selector = B.Selector(shape, sel, DEV)
    out = B.sp_select(selector, w.n_vis, w.n_txt, H=B.dev_f32(H, DEV), stop_bias=B.dev_f32(biases, DEV),
                      group_size=w.group_size, g=w.g, k_max=w.k_max, memory=True)
    torch.cuda.synchronize()
    assert int(out["err"].item()) == 0
    gpu = {k: np_(out[k]) for k in ("order", "ep_count", "rounds", "margin", "gap", "idx", "count")}
    np.testing.assert_array_equal(np_(out["memory"]), H)
    images = PT.oracle_select(H, w.n_vis, sel, k_max=w.k_max, g=w.g, group_size=w.group_size, biases=biases)
    replay, eps_list = PT.replayer(H, w.n_vis, sel, k_max=w.k_max, g=w.g, group_size=w.group_size, biases=biases)
    report = []
    near = PT.compare_selection(gpu, images, g=w.g, report=report, replay=replay, episodes=eps_list)
    for r in report:
        print("near-tie:", r)
    # invariants that hold whatever the ties did
    for b, n in enumerate(w.n_vis):
        k = int(gpu["count"][b])
        row = gpu["idx"][b][:k]
        assert np.all(np.diff(row) > 0) and (k == 0 or (row[0] >= 0 and row[-1] < n))
    selector.close()
    return gpu, images, near


def test_select_tiny_ragged(B):
    w = S.tiny_workload(21, [37, 5, 130, 1, 64], [3, 0, 2, 1, 4], D=128, h=128, k_max=12)
    _run_select_case(B, w, scale=4.0)


def test_select_tiny_stop_extremes(B):
    w = S.tiny_workload(22, [9, 20, 3], [1, 1, 1], D=128, h=128, k_max=8)
    gpu, images, _ = _run_select_case(B, w, scale=4.0, targets=[0, 8, 3])
    assert int(gpu["count"][0]) == 0
    assert int(gpu["count"][1]) == 8 and int(gpu["rounds"][1]) == 8  # cap: no extra round
    assert int(gpu["count"][2]) == 3 and int(gpu["rounds"][2]) == 4  # exhausted: only STOP left


def test_select_max_batch(B):
    # SP_MAX_BATCH images of 1..40 candidates, text 0..3, cap 8
    n_vis = [int(v) for v in S.uniform_int(24, "nv", 1, 41, 256)]
    n_txt = [int(v) for v in S.uniform_int(24, "nt", 0, 4, 256)]
    w = S.tiny_workload(24, n_vis, n_txt, D=128, h=128, k_max=8)
    _run_select_case(B, w, scale=4.0)


def test_select_groups_g5(B):
    w = S.tiny_workload(23, [300, 77, 128], [2, 2, 2], D=128, h=128, k_max=20, group_size=128, g=5)
    _run_select_case(B, w, scale=4.0)


def test_select_llava15_576(B):
    """576 candidates, D=1024, h=256, cap 192 (the single-image workload)."""
    w = S.llava15_1layer()
    _run_select_case(B, w, targets=[64])


def test_select_llava15_b16_full(B):
    """16 x 576 candidates, D=1024, h=512, cap 192, per-image targets 16..192 (mean 64)."""
    w = S.llava15_7b_b16()
    gpu, images, near = _run_select_case(B, w, targets=S.target_counts(w), mean_target=w.target_mean_k)
    counts = gpu["count"].astype(int)
    print("kept counts", counts.tolist(), "mean", counts.mean(), "near-tie episodes", near)


def test_select_anyres_groups(B):
    """8 x 2880 candidates in groups of 576, g=5, per-group cap 128."""
    w = S.llavanext_anyres_b8()
    _run_select_case(B, w, targets=S.uniform_int(w.seed, "t", 16, 129, 40))


def test_select_qwen_varres_cluster16(B):
    """Variable image sizes, D=3584, groups of 1024 (16-CTA clusters hold the keys)."""
    w = S.qwen25vl_varres_b8()
    E = len(PT.episodes(w.n_vis, w.group_size))
    t = [max(1, int(0.11 * n)) for (_, _, n) in PT.episodes(w.n_vis, w.group_size)]
    _run_select_case(B, w, targets=t)


def test_select_internvl_single_episode(B):
    """One episode over 3328 candidates with cap 1024 and g=5 (keys streamed from L2)."""
    w = S.internvl3_tiles_b4(mean_k=128)
    w.n_vis = w.n_vis[:2]
    w.n_txt = w.n_txt[:2]
    _run_select_case(B, w, targets=[128, 512])


# ------------------------------------------------------------------ cross-modal encoder (Eq. 3)

@pytest.mark.parametrize("case", ["tiny", "llava15"])
def test_encoder_memory(B, case):
    if case == "tiny":
        w = S.tiny_workload(31, [40, 130], [7, 0], D=128, D_text=128, h=128, enc_head_dim=64)
    else:
        w = S.llava15_1layer()
    s = w.selector
    sel = S.make_selector_weights(w, ln_affine=True)
    inp = S.make_inputs(w)
    selector = B.Selector(s, sel, DEV)
    E = PT.episodes(w.n_vis, w.group_size)
    out = B.sp_select(selector, w.n_vis, w.n_txt, X=B.dev_bf16(inp["X"], DEV), E_text=B.dev_bf16(inp["E_text"], DEV),
                      stop_bias=B.dev_f32(np.zeros(len(E)), DEV), group_size=0, g=1, k_max=4, memory=True)
    torch.cuda.synchronize()
    got = np_(out["memory"])
    v0 = t0 = 0
    for b in range(w.B):
        Et = O.text_projection(inp["E_text"][t0:t0 + w.n_txt[b]], sel, s.ln_eps, s.g_text)
        ref = O.encoder(inp["X"][v0:v0 + w.n_vis[b]], Et, sel, s.enc_heads, s.ln_eps, store="bf16")
        ref64 = O.encoder(inp["X"][v0:v0 + w.n_vis[b]], Et, sel, s.enc_heads, s.ln_eps)
        g_ = got[v0:v0 + w.n_vis[b]]
        rel = np.abs(g_ - ref).max() / np.sqrt((ref ** 2).mean())
        mrel64 = np.abs(g_ - ref64).mean() / np.abs(ref64).mean()
        print(f"encoder {case} image {b}: vs bf16-storage oracle max-abs / rms {rel:.3e}, vs fp64 mean-rel {mrel64:.3e}")
        assert rel <= PT.HID_MAX_ABS, (b, rel)
        assert mrel64 <= PT.HID_MEAN_REL, (b, mrel64)
        v0 += w.n_vis[b]
        t0 += w.n_txt[b]
    selector.close()


# ------------------------------------------------------------------ compaction (Alg. 1 step 5)

@pytest.mark.parametrize("projector_mode", [False, True])
def test_compaction_bit_exact(B, projector_mode):
    n_vis, n_txt = [576, 7, 1, 300], [48, 0, 5, 13]
    W = 1024
    X = S.bf16_round(S.normal(41, "X", (sum(n_vis), W)))
    text = S.bf16_round(S.normal(41, "T", (sum(n_txt), W)))
    k_cap = 200
    rng = np.random.default_rng(41)
    idx_list = [np.sort(rng.choice(576, 200, replace=False)), np.arange(7), np.zeros(0, int),
                np.sort(rng.choice(300, 17, replace=False))]
    idx = np.full((4, k_cap), -1, np.int32)
    for b, l in enumerate(idx_list):
        idx[b, :len(l)] = l
    count = np.array([len(l) for l in idx_list], np.int32)
    out = B.sp_compact(n_vis, n_txt, X=B.dev_bf16(X, DEV), text=B.dev_bf16(text, DEV), idx=torch.from_numpy(idx).to(DEV),
                       count=torch.from_numpy(count).to(DEV), k_cap=k_cap, projector_mode=projector_mode)
    torch.cuda.synchronize()
    assert int(out["err"].item()) == 0
    packed, cu, pos = O.compact(X, n_vis, idx_list, text, n_txt)
    T = int(cu[-1])
    np.testing.assert_array_equal(np_(out["cu_seqlens"]), cu)
    np.testing.assert_array_equal(np_(out["pos"])[:T], pos)
    got = np_(out["packed"])[:T]
    if not projector_mode:
        np.testing.assert_array_equal(got, packed)
    else:
        vis_rows = np.concatenate([X[sum(n_vis[:b]):][l] for b, l in enumerate(idx_list)])
        R = len(vis_rows)
        np.testing.assert_array_equal(np_(out["vis_packed"])[:R], vis_rows)
        rmap = np_(out["vis_row_map"])[:R]
        np.testing.assert_array_equal(packed[rmap], vis_rows)
        text_rows = np.setdiff1d(np.arange(T), rmap)
        np.testing.assert_array_equal(got[text_rows], packed[text_rows])
        np.testing.assert_array_equal(np_(out["vis_cu"]), np.concatenate([[0], np.cumsum(count)]))


def test_compaction_max_batch(B):
    # SP_MAX_BATCH images: kept counts 0..n (none, some, all), text 0..3 rows
    rng = np.random.default_rng(42)
    n_vis = [int(v) for v in rng.integers(1, 33, 256)]
    n_txt = [int(v) for v in rng.integers(0, 4, 256)]
    W = 256
    X = S.bf16_round(S.normal(42, "X", (sum(n_vis), W)))
    text = S.bf16_round(S.normal(42, "T", (max(sum(n_txt), 1), W)))
    k_cap = 32
    idx_list = []
    for b, n in enumerate(n_vis):
        k = [0, n, int(rng.integers(0, n + 1))][b % 3]
        idx_list.append(np.sort(rng.choice(n, k, replace=False)))
    idx = np.full((256, k_cap), -1, np.int32)
    for b, l in enumerate(idx_list):
        idx[b, :len(l)] = l
    count = np.array([len(l) for l in idx_list], np.int32)
    out = B.sp_compact(n_vis, n_txt, X=B.dev_bf16(X, DEV), text=B.dev_bf16(text, DEV), idx=torch.from_numpy(idx).to(DEV),
                       count=torch.from_numpy(count).to(DEV), k_cap=k_cap)
    torch.cuda.synchronize()
    assert int(out["err"].item()) == 0
    packed, cu, pos = O.compact(X, n_vis, idx_list, text[:sum(n_txt)], n_txt)
    T = int(cu[-1])
    np.testing.assert_array_equal(np_(out["cu_seqlens"]), cu)
    np.testing.assert_array_equal(np_(out["pos"])[:T], pos)
    np.testing.assert_array_equal(np_(out["packed"])[:T], packed)


# ------------------------------------------------------------------ projector

@pytest.mark.parametrize("kind,rows", [("linear", 300), ("mlp2", 300), ("mlp2", 100)])
def test_projector_scatter(B, kind, rows):
    # rows <= 128: the split-K path (GELU and row-scatter epilogues in the reduce pass)
    w = S.tiny_workload(51, [300], [1], D=1024, d=1024, n_heads=8, n_kv_heads=8, head_dim=128, ffn=1024,
                        n_layers=1, proj_kind=kind)
    w.model.proj_hidden = 2048
    head = S.make_model_head(w)
    L = S.make_layer_weights(w, 0)
    model = B.Model(w.model, [L], head, DEV, max_pos=512)
    vis = S.bf16_round(S.normal(51, "vis", (rows, 1024)))
    T = rows + 50
    rmap = np.random.default_rng(51).permutation(T)[:rows].astype(np.int32)
    packed = torch.zeros((T, 1024), dtype=torch.bfloat16, device=DEV)
    vis_cu = torch.tensor([0, rows], dtype=torch.int32, device=DEV)
    err = B.sp_project(model, vis_packed=B.dev_bf16(vis, DEV), vis_row_map=torch.from_numpy(rmap).to(DEV),
                       vis_cu=vis_cu, packed=packed, rows_cap=rows, B=1)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    ref = O.projector(vis, head)
    got = np_(packed)[rmap]
    tol = 1e-2 * np.abs(ref).max()
    assert np.abs(got - ref).max() <= tol, np.abs(got - ref).max()
    untouched = np.setdiff1d(np.arange(T), rmap)
    assert np.all(np_(packed)[untouched] == 0)
    model.close()


@pytest.mark.parametrize("kind,n_vis,keep,k_cap", [
    ("mlp2", [576, 300, 10, 576], [300, 250, 0, 512], 576),   # 1,062 rows: whole tiles
    ("linear", [576, 300, 10, 576], [60, 7, 10, 33], 576),
    ("mlp2", [60, 7, 10, 40], [32, 7, 1, 30], 32)])            # rows_cap 81: split-K GEMM
def test_projector_gather_equals_compact_then_project(B, kind, n_vis, keep, k_cap):
    """Alg. 1 step 5 folded into the projector's operand load: the index-mode
    compaction (no visual row copied, the source row of each kept row written)
    followed by the projector gathering those rows of X gives the packed buffer
    of the copying compaction + projector bit for bit; the source rows are
    exactly the image offsets plus the kept indices."""
    n_txt = [48, 0, 5, 13]
    D = d = 1024
    w = S.tiny_workload(52, [300], [1], D=D, d=d, n_heads=8, n_kv_heads=8, head_dim=128, ffn=1024, n_layers=1,
                        proj_kind=kind)
    w.model.proj_hidden = 2048
    head = S.make_model_head(w)
    model = B.Model(w.model, [S.make_layer_weights(w, 0)], head, DEV, max_pos=1024)
    X = B.dev_bf16(S.bf16_round(S.normal(52, "X", (sum(n_vis), D))), DEV)
    text = B.dev_bf16(S.bf16_round(S.normal(52, "T", (sum(n_txt), d), 0.02)), DEV)
    rng = np.random.default_rng(52)
    idx = np.full((4, k_cap), -1, np.int32)
    idx_list = []
    for b, (n, k) in enumerate(zip(n_vis, keep)):
        l = np.sort(rng.choice(n, k, replace=False)).astype(np.int32)
        idx[b, :k] = l
        idx_list.append(l)
    idx_d = torch.from_numpy(idx).to(DEV)
    cnt_d = torch.tensor(keep, dtype=torch.int32, device=DEV)
    oc = B.sp_compact(n_vis, n_txt, X=X, text=text, idx=idx_d, count=cnt_d, k_cap=k_cap, projector_mode=True)
    e1 = B.sp_project(model, vis_packed=oc["vis_packed"], vis_row_map=oc["vis_row_map"], vis_cu=oc["vis_cu"],
                      packed=oc["packed"], rows_cap=oc["rows_cap"], B=4)
    oi = B.sp_compact(n_vis, n_txt, X=X, text=text, idx=idx_d, count=cnt_d, k_cap=k_cap, index_mode=True)
    e2 = B.sp_project(model, X=X, vis_src=oi["vis_src"], vis_row_map=oi["vis_row_map"], vis_cu=oi["vis_cu"],
                      packed=oi["packed"], rows_cap=oi["rows_cap"], B=4)
    torch.cuda.synchronize()
    assert int(oc["err"].item()) == 0 and int(oi["err"].item()) == 0 and int(e1.item()) == 0 and int(e2.item()) == 0
    R = sum(keep)
    offs = np.concatenate([[0], np.cumsum(n_vis)])
    want_src = np.concatenate([offs[b] + idx_list[b] for b in range(4)])
    np.testing.assert_array_equal(np_(oi["vis_src"])[:R], want_src)
    np.testing.assert_array_equal(np_(oi["vis_row_map"])[:R], np_(oc["vis_row_map"])[:R])
    np.testing.assert_array_equal(np_(oi["cu_seqlens"]), np_(oc["cu_seqlens"]))
    T = int(np_(oc["cu_seqlens"])[-1])
    np.testing.assert_array_equal(np_(oi["pos"])[:T], np_(oc["pos"])[:T])
    a = oi["packed"][:T].view(torch.int16).cpu().numpy()
    b_ = oc["packed"][:T].view(torch.int16).cpu().numpy()
    np.testing.assert_array_equal(a, b_)
    # and the projected rows are the projector of X's kept rows (the oracle, tolerance as the projector test)
    ref = O.projector(np_(X)[want_src], head)
    got = np_(oi["packed"])[np_(oi["vis_row_map"])[:R]]
    assert np.abs(got - ref).max() <= 1e-2 * np.abs(ref).max()
    model.close()


# ------------------------------------------------------------------ prefill

def _prefill_case(B, w, lens, n_layers, seed_name="packed", affine=True):
    layers = [S.make_layer_weights(w, l, norm_affine=affine) for l in range(n_layers)]
    head = S.make_model_head(w, norm_affine=affine)
    model = B.Model(w.model, layers, head, DEV, max_pos=max(lens) + 8)
    T = int(sum(lens))
    x = S.bf16_round(S.normal(w.seed, seed_name, (T, w.model.d), 0.5))
    cu, pos = PT.lens_cu_pos(lens)
    out = B.sp_prefill(model, x=B.dev_bf16(x, DEV), cu_seqlens=torch.from_numpy(cu.astype(np.int32)).to(DEV),
                       pos=torch.from_numpy(pos.astype(np.int32)).to(DEV), B=len(lens), T_cap=T,
                       max_seqlen_cap=max(lens))
    torch.cuda.synchronize()
    assert int(out["err"].item()) == 0
    got = np_(out["hidden"])[:T]
    ref = O.prefill(x, layers, w.model, cu, pos, head["final_norm"], store="bf16")
    r = PT.hidden_close(got, ref, w.name)
    r64 = PT.mean_rel_only(got, O.prefill(x, layers, w.model, cu, pos, head["final_norm"]), w.name)
    print("prefill", w.name, "vs bf16-storage oracle: max-abs %.3e mean-rel %.3e" % r,
          "| vs fp64 oracle: max-abs %.3e mean-rel %.3e" % r64)
    model.close()


def test_prefill_tiny_gqa_ragged(B):
    w = S.tiny_workload(61, [1], [1], D=128, d=128, n_heads=2, n_kv_heads=1, head_dim=64, ffn=256, n_layers=2)
    _prefill_case(B, w, [5, 130, 1, 64], 2)


def test_prefill_llava15_1layer(B):
    w = S.llava15_1layer()
    _prefill_case(B, w, [96, 33, 200], 1)


def _envelope(name):
    """Stored by tests/golden/bf16_envelope.py from the oracle alone: the drift
    between two exact bf16 emulations on this test's inputs (the reference, and
    one with fp32 accumulation and bf16 attention probabilities)."""
    import json
    import os
    with open(os.path.join(os.path.dirname(__file__), "golden", f"bf16_envelope_llava15_7b_{name}.json")) as f:
        return json.load(f)["bf16_fp32acc_bf16p_vs_bf16_fp64acc"]


# end-to-end multi-layer gates: this multiple of the stored drift between two
# exact bf16 emulations (the GPU's rounding decisions flip against the
# reference's through the same fp32 accumulation and bf16 probabilities as the
# second emulation's, in another order)
ENVELOPE_FACTOR = 1.5


def test_prefill_llama7b_dims_2layers(B):
    """Two Llama-7B-dims layers over ragged sequences.

    * Each layer alone, from the oracle's residual at its depth rounded to the
      bf16 input format, at the stated tolerance (max-abs 3e-2, mean-rel 1e-2).
    * Both layers end to end: rounding decisions at the bf16 storage points
      compound with depth, so two exact bf16 prefills that differ only in
      accumulation precision and the precision of the attention probabilities
      already drift apart (stored by the envelope script for these inputs).
      Max-abs within 1.5x that stored drift, mean-rel within the stated 1e-2."""
    w = S.llava15_7b_b16()
    m = w.model
    lens = [112, 240, 64, 17]
    layers = [S.make_layer_weights(w, l, norm_affine=True) for l in range(2)]
    head = S.make_model_head(w, norm_affine=True)
    T = int(sum(lens))
    x = S.bf16_round(S.normal(w.seed, "packed", (T, m.d), 0.5))
    cu, pos = PT.lens_cu_pos(lens)
    cu_d = torch.from_numpy(cu.astype(np.int32)).to(DEV)
    pos_d = torch.from_numpy(pos.astype(np.int32)).to(DEV)

    def gpu(layer_list, inp):
        model = B.Model(m, layer_list, head, DEV, max_pos=max(lens) + 8)
        out = B.sp_prefill(model, x=B.dev_bf16(inp, DEV), cu_seqlens=cu_d, pos=pos_d, B=len(lens), T_cap=T,
                           max_seqlen_cap=max(lens))
        torch.cuda.synchronize()
        assert int(out["err"].item()) == 0
        got = np_(out["hidden"])[:T]
        model.close()
        return got

    # layer-local
    h = x.astype(np.float64)
    for l, L in enumerate(layers):
        xin = S.bf16_round(h.astype(np.float32)).astype(np.float64)
        ref = O.final_norm(O.prefill_layer(xin, L, m, cu, pos, store="bf16"), m, head["final_norm"])
        r = PT.hidden_close(gpu([L], xin.astype(np.float32)), ref, f"layer {l}")
        print(f"layer-local parity, layer {l}: max-abs %.3e mean-rel %.3e" % r)
        h = O.prefill_layer(h, L, m, cu, pos, store="bf16")
    # end to end
    ref = O.prefill(x, layers, m, cu, pos, head["final_norm"], store="bf16")
    ref64 = O.prefill(x, layers, m, cu, pos, head["final_norm"])
    got = gpu(layers, x)
    d = np.abs(got - ref)
    mx, mr = float(d.max()), float(d.mean() / np.abs(ref).mean())
    bound = ENVELOPE_FACTOR * _envelope("2layers")["max_abs"]
    d64 = np.abs(got - ref64)
    print(f"2-layer prefill: vs bf16-storage oracle max-abs {mx:.3e} (bound {bound:.3e}) mean-rel {mr:.3e} | "
          f"vs fp64 oracle max-abs {d64.max():.3e} mean-rel {d64.mean() / np.abs(ref64).mean():.3e}")
    assert mx <= bound and mr <= PT.HID_MEAN_REL, (mx, bound, mr)


def test_prefill_short_batch_split_k(B):
    # T <= 128 packed rows: the GEMMs split K over the SMs and reduce the partials
    # with the fused epilogues (RoPE, residual, SwiGLU) in a second pass
    _prefill_case(B, S.llava15_7b_b16(), [40, 7, 60], 1)
    w = S.tiny_workload(63, [1], [1], D=128, d=128, n_heads=2, n_kv_heads=1, head_dim=64, ffn=256, n_layers=2)
    _prefill_case(B, w, [5, 30, 1, 64], 2)


def test_prefill_empty_sequences(B):
    # zero-length sequences between non-empty ones (repeated cu_seqlens entries)
    w = S.tiny_workload(64, [1], [1], D=128, d=128, n_heads=4, n_kv_heads=2, head_dim=64, ffn=256, n_layers=2)
    _prefill_case(B, w, [0, 5, 0, 130, 1, 0], 2)


def test_prefill_long_with_empty_and_single_token_sequences(B):
    # above 1,280 tokens the two-stream attention kernel runs: zero-length and
    # one-token sequences share its item list with a long one (ragged last
    # tile, GQA 4 / 2, head dim 64); two layers, so the second launch relies on
    # the first leaving the work-ticket counter zero
    w = S.tiny_workload(65, [1], [1], D=128, d=128, n_heads=4, n_kv_heads=2, head_dim=64, ffn=256, n_layers=2)
    _prefill_case(B, w, [0, 1300, 1, 0, 5], 2)


@pytest.mark.parametrize("n", [1280, 1281])
def test_prefill_at_the_attention_kernel_switch(B, n):
    # the longest sequence the call allows picks the attention kernel: 1,280
    # tokens the head-pair kernel, 1,281 the two-stream one (a one-row last tile)
    w = S.tiny_workload(66, [1], [1], D=128, d=128, n_heads=4, n_kv_heads=2, head_dim=64, ffn=256, n_layers=1)
    _prefill_case(B, w, [n, 3], 1)


def test_prefill_qwen_gqa_dims(B):
    w = S.qwen25vl_varres_b8()
    _prefill_case(B, w, [75, 300], 1)


# ------------------------------------------------------------------ whole path

def test_pipeline_end_to_end_without_encoder(B):
    """Selection straight on the visual tokens (no encoder blocks) so that the
    selection is exact end to end; then compaction, projector and prefill."""
    w = S.tiny_workload(71, [200, 64, 130], [9, 3, 0], D=128, D_text=256, h=128, d=256, n_heads=4,
                        n_kv_heads=2, head_dim=64, ffn=256, n_layers=2, k_max=40, proj_kind="mlp2")
    w.model.proj_hidden = 256
    s = w.selector
    sel = S.make_selector_weights(w, ln_affine=True)
    PT.scale_decoder(sel, 4.0)
    sel["enc"] = []
    inp = S.make_inputs(w)
    X, E = inp["X"], inp["E_text"]
    biases = PT.calibrate_biases(X, w.n_vis, sel, k_max=w.k_max, g=1, group_size=0, targets=[17, 40, 5])
    layers = [S.make_layer_weights(w, l, norm_affine=True) for l in range(2)]
    head = S.make_model_head(w, norm_affine=True)
    shape = S.SelectorShape(D=s.D, D_text=s.D_text, h=s.h, n_enc_layers=0)
    selector = B.Selector(shape, sel, DEV)
    model = B.Model(w.model, layers, head, DEV, max_pos=512)
    pipe = B.Pipeline(selector, model, w.n_vis, w.n_txt, group_size=0, g=1, k_max=w.k_max)
    Xd, Ed, bd = B.dev_bf16(X, DEV), B.dev_bf16(E, DEV), B.dev_f32(biases, DEV)
    pipe(Xd, Ed, bd)
    torch.cuda.synchronize()
    assert int(pipe.err.item()) == 0
    ref = O.run_pipeline(X, E, w.n_vis, w.n_txt, sel, shape, head, layers, w.model, k_max=w.k_max, g=1,
                         group_size=0, stop_bias=biases, store="bf16")
    counts = np_(pipe.count)
    for b in range(w.B):
        assert list(np_(pipe.idx)[b][:counts[b]]) == list(ref["idx"][b])
    cu = np_(pipe.cu)
    np.testing.assert_array_equal(cu, ref["cu_seqlens"])
    T = int(cu[-1])
    PT.hidden_close(np_(pipe.hidden)[:T], ref["hidden"], "pipeline")
    # the same call from host buffers gives the same bytes
    Xh, Eh = Xd.cpu().pin_memory(), Ed.cpu().pin_memory()
    bh = bd.cpu().pin_memory()
    oi = torch.empty_like(pipe.idx, device="cpu").pin_memory()
    oc = torch.empty_like(pipe.count, device="cpu").pin_memory()
    ocu = torch.empty_like(pipe.cu, device="cpu").pin_memory()
    oh = torch.empty_like(pipe.hidden, device="cpu").pin_memory()
    pipe.host(Xh, Eh, bh, oi, oc, ocu, oh)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(oi.numpy(), np_(pipe.idx))
    np.testing.assert_array_equal(ocu.numpy(), cu)
    np.testing.assert_array_equal(oh.numpy()[:T], np_(pipe.hidden)[:T])
    # the call is capture-safe (no host synchronisation, sizes from caps): a
    # CUDA graph of it replays to the same bytes
    ref_idx, ref_h = pipe.idx.clone(), pipe.hidden.clone()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        pipe(Xd, Ed, bd)
    pipe.idx.fill_(-7)
    pipe.hidden.zero_()
    pipe.cu.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(pipe.idx, ref_idx)
    np.testing.assert_array_equal(np_(pipe.cu), cu)
    assert torch.equal(pipe.hidden[:T], ref_h[:T])
    selector.close()
    model.close()


def test_pipeline_groups_g5_without_encoder(B):
    """sp_pipeline with candidate groups of 64 and five tokens per round (the
    AnyRes / Qwen / InternVL form), selection straight on the visual tokens so
    that it is exact end to end: indices, offsets and hidden states against the
    oracle's whole path."""
    w = S.tiny_workload(73, [200, 64, 130], [9, 3, 5], D=128, D_text=256, h=128, d=256, n_heads=4,
                        n_kv_heads=2, head_dim=64, ffn=256, n_layers=2, k_max=20, proj_kind="mlp2",
                        group_size=64, g=5)
    w.model.proj_hidden = 256
    s = w.selector
    sel = S.make_selector_weights(w, ln_affine=True)
    PT.scale_decoder(sel, 4.0)
    sel["enc"] = []
    inp = S.make_inputs(w)
    X, E = inp["X"], inp["E_text"]
    # episodes: 64, 64, 64, 8 | 64 | 64, 64, 2 candidates
    biases = PT.calibrate_biases(X, w.n_vis, sel, k_max=w.k_max, g=w.g, group_size=w.group_size,
                                 targets=[10, 20, 5, 8, 15, 20, 10, 2])
    layers = [S.make_layer_weights(w, l, norm_affine=True) for l in range(2)]
    head = S.make_model_head(w, norm_affine=True)
    shape = S.SelectorShape(D=s.D, D_text=s.D_text, h=s.h, n_enc_layers=0)
    selector = B.Selector(shape, sel, DEV)
    model = B.Model(w.model, layers, head, DEV, max_pos=512)
    pipe = B.Pipeline(selector, model, w.n_vis, w.n_txt, group_size=w.group_size, g=w.g, k_max=w.k_max)
    pipe(B.dev_bf16(X, DEV), B.dev_bf16(E, DEV), B.dev_f32(biases, DEV))
    torch.cuda.synchronize()
    assert int(pipe.err.item()) == 0
    ref = O.run_pipeline(X, E, w.n_vis, w.n_txt, sel, shape, head, layers, w.model, k_max=w.k_max, g=w.g,
                         group_size=w.group_size, stop_bias=biases, store="bf16")
    counts = np_(pipe.count)
    for b in range(w.B):
        assert list(np_(pipe.idx)[b][:counts[b]]) == list(ref["idx"][b])
    cu = np_(pipe.cu)
    np.testing.assert_array_equal(cu, ref["cu_seqlens"])
    T = int(cu[-1])
    r = PT.hidden_close(np_(pipe.hidden)[:T], ref["hidden"], "grouped pipeline")
    print("grouped g=5 pipeline: kept", counts.tolist(), "max-abs %.3e mean-rel %.3e" % r)
    selector.close()
    model.close()


def test_pipeline_with_encoder_equals_its_stages(B):
    """The chained call with the 2-block encoder, candidate groups and g = 5
    gives the bytes of its stages called one by one through the C ABI
    (sp_select -> sp_compact (index mode) -> sp_project -> sp_prefill), each
    of which is compared with the oracle on its own."""
    w = S.tiny_workload(74, [200, 64, 130], [9, 3, 5], D=128, D_text=256, h=128, d=256, n_heads=4,
                        n_kv_heads=2, head_dim=64, ffn=256, n_layers=2, k_max=20, proj_kind="mlp2",
                        group_size=64, g=5, enc_head_dim=64)
    w.model.proj_hidden = 256
    sel = S.make_selector_weights(w, ln_affine=True)
    inp = S.make_inputs(w)
    layers = [S.make_layer_weights(w, l, norm_affine=True) for l in range(2)]
    head = S.make_model_head(w, norm_affine=True)
    selector = B.Selector(w.selector, sel, DEV)
    model = B.Model(w.model, layers, head, DEV, max_pos=512)
    Xd, Ed = B.dev_bf16(inp["X"], DEV), B.dev_bf16(inp["E_text"], DEV)
    n_ep = len(w.episodes())
    # a STOP bias far below / above the logits keeps each group to k_max / stops it at once
    assert n_ep == 8  # 64, 64, 64, 8 | 64 | 64, 64, 2 candidates
    bd = B.dev_f32(np.array([-1.5, 1.5, -1.5, 1.5, -1.5, 1.5, -1.5, -1.5], np.float32), DEV)
    pipe = B.Pipeline(selector, model, w.n_vis, w.n_txt, group_size=w.group_size, g=w.g, k_max=w.k_max)
    pipe(Xd, Ed, bd)
    r = B.sp_select(selector, w.n_vis, w.n_txt, X=Xd, E_text=Ed, stop_bias=bd, group_size=w.group_size, g=w.g,
                    k_max=w.k_max, k_cap=pipe.k_cap, traces=False)
    c = B.sp_compact(w.n_vis, w.n_txt, X=Xd, text=Ed, idx=r["idx"], count=r["count"], k_cap=pipe.k_cap,
                     index_mode=True)
    B.sp_project(model, vis_row_map=c["vis_row_map"], vis_cu=c["vis_cu"], packed=c["packed"],
                 rows_cap=c["rows_cap"], B=w.B, X=Xd, vis_src=c["vis_src"])
    max_len = max(min(n, pipe.k_cap) + t for n, t in zip(w.n_vis, w.n_txt))
    p = B.sp_prefill(model, x=c["packed"], cu_seqlens=c["cu_seqlens"], pos=c["pos"], B=w.B, T_cap=c["T_cap"],
                     max_seqlen_cap=max_len)
    torch.cuda.synchronize()
    assert int(pipe.err.item()) == 0 and int(c["err"].item()) == 0 and int(p["err"].item()) == 0
    counts = np_(pipe.count)
    assert counts.tolist() == np_(r["count"]).tolist() and 0 < counts.sum() < sum(w.n_vis)
    np.testing.assert_array_equal(np_(pipe.idx), np_(r["idx"]))
    cu = np_(pipe.cu)
    np.testing.assert_array_equal(cu, np_(c["cu_seqlens"]))
    T = int(cu[-1])
    np.testing.assert_array_equal(np_(pipe.hidden)[:T], np_(p["hidden"])[:T])
    print("pipeline with encoder: kept", counts.tolist(), "of", w.n_vis)
    selector.close()
    model.close()


def test_prefill_llava15_b16_32layers_sampled(B):
    """The benchmark's prefill launch: 32 Llama-7B-dims layers over 16 packed
    sequences (kept counts 16..192 + 48 text tokens).

    * Layer-local parity (the stated tolerance, max-abs 3e-2 / mean-rel 1e-2):
      layers 0, 15 and 31 run alone on the GPU from the oracle's own residual at
      that depth (rounded to the bf16 input format), against the oracle layer.
    * End to end over 32 layers, on two sampled sequences (the shortest and the
      longest; attention never crosses a sequence, so their rows are exact to
      compare): the stated 3e-2 / 1e-2 does not hold at this depth for any bf16
      prefill (a known miss): two exact bf16 emulations that differ only in
      accumulation precision and the precision of the attention probabilities
      drift apart by the stored envelope; max-abs and mean-rel within 1.5x that
      envelope."""
    import dataclasses
    w = S.llava15_7b_b16()
    m = dataclasses.replace(w.model, proj_kind="none", proj_in=w.model.d)
    k = S.target_counts(w)
    lens = [int(x) + 48 for x in k]
    T = sum(lens)
    cu, pos = PT.lens_cu_pos(lens)
    x = S.bf16_round(S.normal(w.seed, "packed32", (T, m.d), 0.5))
    picks = [int(np.argmin(lens)), int(np.argmax(lens))]
    hs = {b: x[cu[b]:cu[b + 1]].astype(np.float64) for b in picks}
    local_layers = (0, 15, 31)
    local = {}
    dev_layers = []
    for l in range(m.n_layers):
        L = S.make_layer_weights(w, l)
        dev_layers.append({k_: B.dev_bf16(L[k_], DEV) for k_ in ("Wqkv", "Wo", "Wgu", "Wdown")})
        dev_layers[-1]["attn_norm"] = torch.ones(m.d, device=DEV)
        dev_layers[-1]["mlp_norm"] = torch.ones(m.d, device=DEV)
        if l in local_layers:
            xin = {b: S.bf16_round(hs[b].astype(np.float32)).astype(np.float64) for b in picks}
            ref = {b: O.final_norm(O.prefill_layer(xin[b], L, m, [0, lens[b]], np.arange(lens[b]), store="bf16"), m)
                   for b in picks}
            local[l] = (xin, ref)
        for b in picks:
            n = lens[b]
            hs[b] = O.prefill_layer(hs[b], L, m, [0, n], np.arange(n), store="bf16")
        del L
    head = {"final_norm": torch.ones(m.d, device=DEV), "proj_W1": None, "proj_W2": None}
    model = B.Model(m, None, None, DEV, max_pos=512, device_weights={"layers": dev_layers, "head": head})
    out = B.sp_prefill(model, x=B.dev_bf16(x, DEV), cu_seqlens=torch.from_numpy(cu.astype(np.int32)).to(DEV),
                       pos=torch.from_numpy(pos.astype(np.int32)).to(DEV), B=len(lens), T_cap=T,
                       max_seqlen_cap=max(lens))
    torch.cuda.synchronize()
    assert int(out["err"].item()) == 0
    got = np_(out["hidden"])
    env = _envelope("32layers")
    g_all = np.concatenate([got[cu[b]:cu[b + 1]] for b in picks])
    r_all = np.concatenate([O.final_norm(hs[b], m) for b in picks])
    d = np.abs(g_all - r_all)
    mx, mr = float(d.max()), float(d.mean() / np.abs(r_all).mean())
    print(f"32-layer prefill, sequences {picks} (lens {[lens[b] for b in picks]}): max-abs {mx:.3e} mean-rel {mr:.3e} "
          f"(bounds {ENVELOPE_FACTOR * env['max_abs']:.3e} / {ENVELOPE_FACTOR * env['mean_rel']:.3e})")
    assert mx <= ENVELOPE_FACTOR * env["max_abs"] and mr <= ENVELOPE_FACTOR * env["mean_rel"], (mx, mr)
    model.close()
    # layer-local parity at the stated tolerance
    sub = [lens[b] for b in picks]
    cu2, pos2 = PT.lens_cu_pos(sub)
    for l in local_layers:
        one = B.Model(m, None, None, DEV, max_pos=512,
                      device_weights={"layers": [dev_layers[l]], "head": head})
        xin, ref = local[l]
        xx = np.concatenate([xin[b] for b in picks]).astype(np.float32)
        o = B.sp_prefill(one, x=B.dev_bf16(xx, DEV), cu_seqlens=torch.from_numpy(cu2.astype(np.int32)).to(DEV),
                         pos=torch.from_numpy(pos2.astype(np.int32)).to(DEV), B=2, T_cap=int(cu2[-1]),
                         max_seqlen_cap=max(sub))
        torch.cuda.synchronize()
        g2 = np_(o["hidden"])
        r = PT.hidden_close(g2, np.concatenate([ref[b] for b in picks]), f"layer {l}")
        print(f"layer-local parity, layer {l}: max-abs %.3e mean-rel %.3e" % r)
        one.close()


# ------------------------------------------------------------------ generation over the pruned prefix

def _decode_case(B, w, lens, n_layers, steps=2):
    """The prefill's cache (parity of every cached row against the oracle's),
    then generation steps: the first fed the oracle's own cache (stage-local),
    the next chained on the GPU's cache."""
    m = w.model
    layers = [S.make_layer_weights(w, l, norm_affine=True) for l in range(n_layers)]
    head = S.make_model_head(w, norm_affine=True)
    model = B.Model(m, layers, head, DEV, max_pos=max(lens) + steps + 8)
    T = int(sum(lens))
    nb = len(lens)
    x = S.bf16_round(S.normal(w.seed, "packed", (T, m.d), 0.5))
    cu, pos = PT.lens_cu_pos(lens)
    S_cap = max(lens) + steps
    kv_rows = []
    O.prefill(x, layers, m, cu, pos, head["final_norm"], store="bf16", kv_out=kv_rows)
    cache = O.cache_from_prefill(kv_rows, cu)

    # prefill writes the cache
    kv = B.kv_cache(model, nb, S_cap)
    out = B.sp_prefill(model, x=B.dev_bf16(x, DEV), cu_seqlens=torch.from_numpy(cu.astype(np.int32)).to(DEV),
                       pos=torch.from_numpy(pos.astype(np.int32)).to(DEV), B=nb, T_cap=T, max_seqlen_cap=max(lens),
                       kv=kv)
    torch.cuda.synchronize()
    assert int(out["err"].item()) == 0
    got_kv = kv.float().cpu().numpy()
    for l in range(n_layers):
        for b in range(nb):
            for j, name in ((0, "K"), (1, "V")):
                if lens[b] == 0:
                    continue
                ref = cache[l][b][j]
                g = got_kv[l, j, b, :lens[b]]
                err = np.abs(g - ref).max() / max(np.abs(ref).max(), 1e-6)
                # layer 0 is one GEMM from the same bf16 input: one rounding flip at most
                bound = 1e-2 if l == 0 else 5e-2
                assert err <= bound, (l, b, name, err)
            assert np.all(got_kv[l, :, b, lens[b]:] == 0)  # positions past the prefix untouched

    # step 1 from the oracle's cache, then chained steps on the GPU cache
    kv_o = B.kv_cache(model, nb, S_cap)
    host = kv_o.float().cpu().numpy()
    for l in range(n_layers):
        for b in range(nb):
            host[l, 0, b, :lens[b]] = cache[l][b][0]
            host[l, 1, b, :lens[b]] = cache[l][b][1]
    kv_o.copy_(torch.from_numpy(host).to(torch.bfloat16))
    lens_d = torch.tensor(lens, dtype=torch.int32, device=DEV)
    ws = None
    for step in range(steps):
        x_new = S.bf16_round(S.normal(w.seed, f"new{step}", (nb, m.d), 0.5))
        o = B.sp_decode(model, x=B.dev_bf16(x_new, DEV), lens=lens_d, kv=kv_o, max_len_cap=S_cap, ws=ws)
        ws = o["_ws"]
        torch.cuda.synchronize()
        assert int(o["err"].item()) == 0
        ref, cache = O.decode_step(x_new, layers, m, cache, head["final_norm"], store="bf16")
        r = PT.hidden_close(np_(o["hidden"]), ref, f"{w.name} decode step {step}")
        print(f"decode step {step}: max-abs %.3e mean-rel %.3e" % r)
        np.testing.assert_array_equal(lens_d.cpu().numpy(), np.array(lens) + step + 1)
    model.close()


def test_decode_steps_replay_in_a_cuda_graph(B):
    """A generation step is capture-safe (lengths live and advance on the
    device, no host synchronisation): the same steps issued one by one and
    replayed from a captured CUDA graph give the same bits, hidden states and
    cache alike (Llama-7B dims, one layer, weight-streaming GEMMs)."""
    w = S.llava15_7b_b16()
    m = w.model
    L = S.make_layer_weights(w, 0, norm_affine=True)
    head = S.make_model_head(w, norm_affine=True)
    model = B.Model(m, [L], head, DEV, max_pos=512)
    lens = [112, 240, 64, 17]
    nb, steps = len(lens), 3
    S_cap = max(lens) + steps + 8
    x_new = B.dev_bf16(S.bf16_round(S.normal(w.seed, "decode_graph", (nb, m.d), 0.5)), DEV)
    rng = np.random.default_rng(5)
    init = (torch.from_numpy(rng.standard_normal((1, 2, nb, S_cap, m.n_kv_heads * m.head_dim)).astype(np.float32))
            .to(torch.bfloat16).to(DEV))
    runs = []
    for graph in (False, True):
        kv = init.clone()
        lens_d = torch.tensor(lens, dtype=torch.int32, device=DEV)
        hid = torch.zeros((nb, m.d), dtype=torch.float32, device=DEV)
        ws = B.sp_decode(model, x=x_new, lens=torch.tensor(lens, dtype=torch.int32, device=DEV), kv=init.clone(),
                         max_len_cap=S_cap, hidden=torch.zeros_like(hid))["_ws"]
        torch.cuda.synchronize()
        step = lambda: B.sp_decode(model, x=x_new, lens=lens_d, kv=kv, max_len_cap=S_cap, ws=ws, hidden=hid)
        outs = []
        if graph:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                step()
            lens_d.copy_(torch.tensor(lens, dtype=torch.int32, device=DEV))  # (capture does not run the step)
            for _ in range(steps):
                g.replay()
                outs.append(hid.clone())
        else:
            for _ in range(steps):
                step()
                outs.append(hid.clone())
        torch.cuda.synchronize()
        runs.append(([o.cpu() for o in outs], kv.cpu(), lens_d.cpu()))
    (h0, kv0, l0), (h1, kv1, l1) = runs
    assert torch.equal(l0, l1) and l0.tolist() == [n + steps for n in lens]
    for a, b in zip(h0, h1):
        assert torch.equal(a, b)
    assert torch.equal(kv0, kv1)
    model.close()


def test_decode_tiny_gqa_ragged(B):
    w = S.tiny_workload(62, [1], [1], D=128, d=128, n_heads=4, n_kv_heads=2, head_dim=64, ffn=256, n_layers=2)
    _decode_case(B, w, [5, 130, 1, 64], 2)


def test_decode_empty_prefix(B):
    # a sequence with no cached positions attends to its new token alone
    w = S.tiny_workload(65, [1], [1], D=128, d=128, n_heads=4, n_kv_heads=2, head_dim=64, ffn=256, n_layers=2)
    _decode_case(B, w, [0, 7, 1], 2)


def test_decode_long_prefix_gqa8(B):
    # 8 query heads per key / value head (the widest group the decode takes) and
    # a prefix longer than 16 key ranges of 64: each range then spans several
    # shared-memory tiles of keys
    w = S.tiny_workload(66, [1], [1], D=128, d=256, n_heads=8, n_kv_heads=1, head_dim=128, ffn=256, n_layers=1)
    _decode_case(B, w, [1300, 65, 0, 64], 1)


def test_decode_llama7b_dims_1layer(B):
    w = S.llava15_7b_b16()
    _decode_case(B, w, [112, 240, 64, 17], 1)


@pytest.mark.parametrize("nb", [16, 32, 33])
def test_decode_llama7b_dims_batch_edges(B, nb):
    # 16 and 32 sequences take the weight-streaming GEMMs (activations as the
    # MMA's 32 columns: one or two 16-row halves), 33 the 128-row-tile path
    w = S.llava15_7b_b16()
    rng = np.random.default_rng(900 + nb)
    lens = [int(v) for v in rng.integers(0, 24, nb)]
    lens[0] = 0
    _decode_case(B, w, lens, 1)
