"""Small, self-contained invocations of one stage of the path, sized for
`ncu --set full` captures (a few GB on the device at most, a handful of
launches).  Shapes are those of the 16-image LLaVA-1.5-7B-shaped batch.

    python -m paper_2609_13804_gb300.profile_case gemm       # 1 decoder layer, T = 1791 (4 GEMMs)
    python -m paper_2609_13804_gb300.profile_case select     # selection from a given memory H
    python -m paper_2609_13804_gb300.profile_case select_deep  # 2-layer pointer decoder, 4 images, cap 64
    python -m paper_2609_13804_gb300.profile_case compact    # compaction of the batch
    python -m paper_2609_13804_gb300.profile_case compact_full  # every visual token kept (50 MB)
    python -m paper_2609_13804_gb300.profile_case attention  # 1 decoder layer, like gemm
    python -m paper_2609_13804_gb300.profile_case attention_full  # 1 layer over the full prefix (16 x 624)
    python -m paper_2609_13804_gb300.profile_case decode     # 4 decoder layers, 16 sequences, 3 steps

Each case runs its stage twice (the second launch set is the one to capture
with `-s`).
"""
import dataclasses
import sys

import numpy as np


def main(case: str):
    import torch

    from paper_2609_13804_gb300 import binding as B
    from paper_2609_13804_gb300 import synth as S

    dev = torch.device("cuda", 0)
    w = S.llava15_7b_b16()
    counts = S.target_counts(w)
    if case in ("gemm", "attention", "attention_full", "decode"):
        m = dataclasses.replace(w.model, proj_kind="none", proj_in=w.model.d)
        gen = torch.Generator(device=dev)
        gen.manual_seed(1)

        def rnd(shape):
            return (torch.randn(shape, device=dev, generator=gen) * 0.02).to(torch.bfloat16)

        qkv = (m.n_heads + 2 * m.n_kv_heads) * m.head_dim
        L = {"Wqkv": rnd((qkv, m.d)), "Wo": rnd((m.d, m.n_heads * m.head_dim)), "Wgu": rnd((2 * m.ffn, m.d)),
             "Wdown": rnd((m.d, m.ffn)), "attn_norm": torch.ones(m.d, device=dev),
             "mlp_norm": torch.ones(m.d, device=dev)}
        head = {"final_norm": torch.ones(m.d, device=dev), "proj_W1": None, "proj_W2": None}
        n_layers = 4 if case == "decode" else 1
        layers = [L] + [{k: (rnd(v.shape) if v.dtype == torch.bfloat16 else v) for k, v in L.items()}
                        for _ in range(n_layers - 1)]
        m = dataclasses.replace(m, n_layers=n_layers)
        model = B.Model(m, None, None, dev, max_pos=1024, device_weights={"layers": layers, "head": head})
        lens = [int(k) + 48 for k in counts]
        if case == "attention_full":
            lens = [n + t for n, t in zip(w.n_vis, w.n_txt)]  # every visual token kept: 624 per sequence
        if case == "decode":
            # one generation step per sequence over the pruned prefix (a zeroed
            # cache with the prefix lengths: the contents do not change the work)
            S_cap = max(lens) + 8
            kv = B.kv_cache(model, len(lens), S_cap)
            x_new = (torch.randn((len(lens), m.d), device=dev, generator=gen) * 0.5).to(torch.bfloat16)
            lens_d = torch.tensor(lens, dtype=torch.int32, device=dev)
            ws = None
            for _ in range(3):
                ws = B.sp_decode(model, x=x_new, lens=lens_d, kv=kv, max_len_cap=S_cap, ws=ws)["_ws"]
            torch.cuda.synchronize()
            print("ok", case)
            return
        T = sum(lens)
        cu = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int32, device=dev)
        pos = torch.tensor(np.concatenate([np.arange(n) for n in lens]), dtype=torch.int32, device=dev)
        x = (torch.randn((T, m.d), device=dev, generator=gen) * 0.5).to(torch.bfloat16)
        # the caps of the pipeline (k_cap 192 per image) so tile widths match the benchmark's launches
        kc = max(w.n_vis) if case == "attention_full" else w.k_max
        T_cap = sum(min(n, kc) + t for n, t in zip(w.n_vis, w.n_txt))
        len_cap = max(min(n, kc) + t for n, t in zip(w.n_vis, w.n_txt))
        xc = torch.zeros((T_cap, m.d), dtype=torch.bfloat16, device=dev)
        xc[:T] = x
        pc = torch.zeros(T_cap, dtype=torch.int32, device=dev)
        pc[:T] = pos
        ws = None
        for _ in range(2):
            out = B.sp_prefill(model, x=xc, cu_seqlens=cu, pos=pc, B=len(lens), T_cap=T_cap, max_seqlen_cap=len_cap,
                               ws=ws)
            ws = out["_ws"]
        torch.cuda.synchronize()
    elif case == "select":
        s = S.SelectorShape(D=w.selector.D, D_text=w.selector.D_text, h=w.selector.h, n_enc_layers=0)
        sel = S.make_selector_weights(w)
        H = S.make_memory(w)
        selector = B.Selector(s, sel, dev)
        Hd = B.dev_f32(H, dev)
        bias = B.dev_f32(np.full(w.B, -1e30), dev)   # every episode runs to its cap of 192
        ws = None
        for _ in range(2):
            r = B.sp_select(selector, w.n_vis, w.n_txt, H=Hd, stop_bias=bias, k_max=w.k_max, traces=False, ws=ws)
            ws = r["_ws"]
        torch.cuda.synchronize()
    elif case == "select_deep":
        w.n_vis, w.n_txt = w.n_vis[:4], w.n_txt[:4]
        s = S.SelectorShape(D=w.selector.D, D_text=w.selector.D_text, h=w.selector.h, n_enc_layers=0,
                            n_dec_layers=2)
        w = dataclasses.replace(w, selector=s)
        selector = B.Selector(s, S.make_selector_weights(w), dev)
        Hd = B.dev_f32(S.make_memory(w), dev)
        bias = B.dev_f32(np.full(4, -1e30), dev)
        ws = None
        for _ in range(2):
            r = B.sp_select(selector, w.n_vis, w.n_txt, H=Hd, stop_bias=bias, k_max=64, traces=False, ws=ws)
            ws = r["_ws"]
        torch.cuda.synchronize()
    elif case == "compact_full":
        # every visual token kept: the bandwidth-sized compaction (50 MB moved)
        X = B.dev_bf16(S.bf16_round(S.normal(w.seed, "X", (sum(w.n_vis), 1024))), dev)
        E = B.dev_bf16(S.bf16_round(S.normal(w.seed, "E", (sum(w.n_txt), 4096), 0.02)), dev)
        idx = torch.arange(576, dtype=torch.int32, device=dev).repeat(w.B, 1).contiguous()
        cnt = torch.full((w.B,), 576, dtype=torch.int32, device=dev)
        for _ in range(2):
            B.sp_compact(w.n_vis, w.n_txt, X=X, text=E, idx=idx, count=cnt, k_cap=576, projector_mode=True)
        torch.cuda.synchronize()
    elif case == "compact":
        X = B.dev_bf16(S.bf16_round(S.normal(w.seed, "X", (sum(w.n_vis), 1024))), dev)
        E = B.dev_bf16(S.bf16_round(S.normal(w.seed, "E", (sum(w.n_txt), 4096), 0.02)), dev)
        k_cap = 192
        idx = torch.full((w.B, k_cap), -1, dtype=torch.int32, device=dev)
        for b, k in enumerate(counts):
            idx[b, :k] = torch.arange(0, 576, 576 // max(int(k), 1), device=dev)[:k].to(torch.int32)
        cnt = torch.tensor(counts, dtype=torch.int32, device=dev)
        for _ in range(2):
            B.sp_compact(w.n_vis, w.n_txt, X=X, text=E, idx=idx, count=cnt, k_cap=k_cap, projector_mode=True)
        torch.cuda.synchronize()
    else:
        raise SystemExit(f"unknown case {case}")
    print("ok", case)


if __name__ == "__main__":
    main(sys.argv[1] if len(sys.argv) > 1 else "gemm")
