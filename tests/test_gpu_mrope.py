"""GPU parity of the 3-D mRoPE variant (the Qwen2.5-VL backbone, Sec. 1):
the packed batch's (t, h, w) positions (bit-exact), the prefill with mRoPE
(the prefill tolerances) and generation after an mRoPE prefix at explicit
rotary positions, each fed seeded inputs and compared with the oracle."""
import dataclasses

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
    return t.float().cpu().numpy() if t.dtype == torch.bfloat16 else t.cpu().numpy()


def _kept(seed, n_vis, counts):
    out = []
    for b, (n, k) in enumerate(zip(n_vis, counts)):
        out.append(np.sort(np.random.default_rng(seed + b).choice(n, size=k, replace=False)).astype(np.int64))
    return out


def _oracle_pos3(kept, n_vis, grid_w, n_txt):
    return np.concatenate([O.mrope_positions(k, n, g, t) for k, n, g, t in zip(kept, n_vis, grid_w, n_txt)])


def test_mrope_positions_bit_exact(B):
    n_vis = [1024, 576, 10, 2304, 7, 256]
    grid_w = [32, 24, 4, 48, 7, 16]          # image 2: a 3 x 4 grid with its last row partly filled
    n_txt = [64, 3, 0, 64, 5, 1]
    counts = [100, 0, 10, 300, 7, 31]        # none, all, ragged
    kept = _kept(7, n_vis, counts)
    k_cap = 320
    idx = np.full((len(n_vis), k_cap), -1, np.int32)
    for b, k in enumerate(kept):
        idx[b, :len(k)] = k
    T = sum(counts) + sum(n_txt)
    r = B.sp_mrope_positions(n_vis, n_txt, grid_w, idx=torch.from_numpy(idx).to(DEV),
                             count=torch.tensor(counts, dtype=torch.int32, device=DEV), k_cap=k_cap, T_cap=T + 5)
    torch.cuda.synchronize()
    assert int(r["err"].item()) == 0
    got = r["pos3"].cpu().numpy()
    want = _oracle_pos3(kept, n_vis, grid_w, n_txt)
    np.testing.assert_array_equal(got[:T, :3], want.astype(np.int32))
    assert np.all(got[T:] == 0)  # rows past the packed length untouched


def test_mrope_positions_flags_bad_indices(B):
    idx = torch.tensor([[0, 3, 99, -1]], dtype=torch.int32, device=DEV)  # 99 is outside the 16-token image
    r = B.sp_mrope_positions([16], [2], [4], idx=idx, count=torch.tensor([3], dtype=torch.int32, device=DEV),
                             k_cap=4, T_cap=5)
    torch.cuda.synchronize()
    assert int(r["err"].item()) != 0
    assert r["pos3"][:2, :3].cpu().numpy().tolist() == [[0, 0, 0], [0, 0, 3]]


def _mrope_prefill(B, w, section, n_vis, grid_w, counts, n_txt, n_layers, seed):
    m = dataclasses.replace(w.model, mrope_section=tuple(section))
    kept = _kept(seed, n_vis, counts)
    pos3 = _oracle_pos3(kept, n_vis, grid_w, n_txt)
    lens = [k + t for k, t in zip(counts, n_txt)]
    layers = [S.make_layer_weights(w, l, norm_affine=True) for l in range(n_layers)]
    head = S.make_model_head(w, norm_affine=True)
    model = B.Model(m, layers, head, DEV, max_pos=max(int(pos3.max()), max(lens)) + 8)
    T = int(sum(lens))
    x = S.bf16_round(S.normal(w.seed, "packed", (T, m.d), 0.5))
    cu, pos = PT.lens_cu_pos(lens)
    p4 = np.zeros((T, 4), np.int32)
    p4[:, :3] = pos3
    out = B.sp_prefill(model, x=B.dev_bf16(x, DEV), cu_seqlens=torch.from_numpy(cu.astype(np.int32)).to(DEV),
                       pos=torch.from_numpy(pos.astype(np.int32)).to(DEV), B=len(lens), T_cap=T,
                       max_seqlen_cap=max(lens), pos3=torch.from_numpy(p4).to(DEV))
    torch.cuda.synchronize()
    assert int(out["err"].item()) == 0
    got = np_(out["hidden"])[:T]
    ref = O.prefill(x, layers, m, cu, pos3, head["final_norm"], store="bf16")
    r = PT.hidden_close(got, ref, w.name + " mrope")
    # the 3-D positions matter: against the same rows under 1-D positions the
    # GPU result is much further off
    ref1 = O.prefill(x, layers, m, cu, pos, head["final_norm"], store="bf16")
    assert np.abs(got - ref1).mean() > 5 * np.abs(got - ref).mean()
    print("mrope prefill", w.name, "max-abs %.3e mean-rel %.3e" % r)
    model.close()


def test_prefill_mrope_tiny_ragged(B):
    w = S.tiny_workload(63, [1], [1], D=128, d=128, n_heads=2, n_kv_heads=1, head_dim=64, ffn=256, n_layers=2)
    _mrope_prefill(B, w, (8, 12, 12), [64, 30, 9], [8, 6, 3], [20, 30, 1], [5, 0, 4], 2, 11)


def test_prefill_mrope_qwen_dims(B):
    w = S.qwen25vl_varres_b8()
    _mrope_prefill(B, w, (16, 24, 24), [1024, 2304], [32, 48], [11, 236], [64, 64], 1, 12)


def test_decode_after_mrope_prefix(B):
    """Generated text tokens after an mRoPE prefix: the cache from the oracle's
    prefill, two steps at explicit rotary positions (incremented on the device)."""
    w = S.tiny_workload(64, [1], [1], D=128, d=128, n_heads=4, n_kv_heads=2, head_dim=64, ffn=256, n_layers=2)
    m = dataclasses.replace(w.model, mrope_section=(8, 12, 12))
    n_vis, grid_w, counts, n_txt = [64, 30], [8, 6], [20, 30], [5, 3]
    kept = _kept(13, n_vis, counts)
    pos3 = _oracle_pos3(kept, n_vis, grid_w, n_txt)
    lens = [k + t for k, t in zip(counts, n_txt)]
    nb, steps = len(lens), 2
    layers = [S.make_layer_weights(w, l, norm_affine=True) for l in range(2)]
    head = S.make_model_head(w, norm_affine=True)
    S_cap = max(lens) + steps
    model = B.Model(m, layers, head, DEV, max_pos=int(pos3.max()) + steps + 1)  # below max(lens): fine with rope_pos
    T = int(sum(lens))
    x = S.bf16_round(S.normal(w.seed, "packed", (T, m.d), 0.5))
    cu, _ = PT.lens_cu_pos(lens)
    kv_rows = []
    O.prefill(x, layers, m, cu, pos3, head["final_norm"], store="bf16", kv_out=kv_rows)
    cache = O.cache_from_prefill(kv_rows, cu)
    kv = B.kv_cache(model, nb, S_cap)
    host = kv.float().cpu().numpy()
    for l in range(2):
        for b in range(nb):
            host[l, 0, b, :lens[b]] = cache[l][b][0]
            host[l, 1, b, :lens[b]] = cache[l][b][1]
    kv.copy_(torch.from_numpy(host).to(torch.bfloat16))
    lens_d = torch.tensor(lens, dtype=torch.int32, device=DEV)
    nxt = [int(pos3[cu[b + 1] - 1, 0]) + 1 for b in range(nb)]
    rp = torch.tensor(nxt, dtype=torch.int32, device=DEV)
    ws = None
    for step in range(steps):
        x_new = S.bf16_round(S.normal(w.seed, f"new{step}", (nb, m.d), 0.5))
        o = B.sp_decode(model, x=B.dev_bf16(x_new, DEV), lens=lens_d, kv=kv, max_len_cap=S_cap, ws=ws, rope_pos=rp)
        ws = o["_ws"]
        torch.cuda.synchronize()
        assert int(o["err"].item()) == 0
        ref, cache = O.decode_step(x_new, layers, m, cache, head["final_norm"], store="bf16",
                                   rope_pos=[p + step for p in nxt])
        r = PT.hidden_close(np_(o["hidden"]), ref, f"mrope decode step {step}")
        print(f"mrope decode step {step}: max-abs %.3e mean-rel %.3e" % r)
        np.testing.assert_array_equal(rp.cpu().numpy(), np.array(nxt) + step + 1)
        np.testing.assert_array_equal(lens_d.cpu().numpy(), np.array(lens) + step + 1)
    model.close()
