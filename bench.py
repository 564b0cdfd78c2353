"""Benchmark of the StepPrune inference path on the LLaVA-1.5-7B-shaped batch.

One step = one sp_pipeline call over a batch of 16 images x 576 visual tokens
(+ 48 text tokens each): text projection and the 2-block cross-modal encoder,
candidate precompute, the sequential selection loop, restore, compaction, the
2-layer GELU projector on the kept rows and the 32-layer Llama-7B-dims prefill
over the packed prefix.  Random-init weights and seeded synthetic inputs; STOP
biases tuned so the kept counts span 16..192 with mean about 64.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line (rank 0).  `value` is ms per batch over the whole job
(lower is better); with N ranks each rank runs its own batch (weak scaling).
`--impl reference` times the CPU oracle on a bounded sample of the same
workload instead.
"""
import argparse
import dataclasses
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2609_13804_gb300 import synth as S  # noqa: E402
from paper_2609_13804_gb300.replicas import max_over_ranks  # noqa: E402

METRIC = "pruned-prefill ms/batch"
UNIT = "ms/batch"


# DRAM read + write bytes per prefill GEMM launch (mean over QKV, O, gate/up and
# down) from the ncu capture summarised in profiles/gemm_tc2_llava15-7b-dims_1layer.md
# (one 7B-dims layer at T = 1,792 rows, the benchmark's packed length within
# 0.5%).  The figure belongs to the kernel sources with this digest; once they
# change it is reported as null until a new capture replaces it.
GEMM_TRAFFIC = {"bytes_per_launch": 163.7e6, "sources_sha256_16": "b9fa2d347c9187a4"}
GEMM_SOURCES = ("paper_2609_13804_gb300/csrc/gemm_tc.cu", "paper_2609_13804_gb300/csrc/common.cuh")


def gemm_traffic():
    import hashlib
    h = hashlib.sha256()
    for rel in GEMM_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return GEMM_TRAFFIC["bytes_per_launch"] if h.hexdigest()[:16] == GEMM_TRAFFIC["sources_sha256_16"] else None


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16": d["bf16_tflops"], "bf16_sus": d["bf16_tflops_sustained"],
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16": 1900.0, "bf16_sus": 1700.0, "source": "fallback"}


# ----------------------------------------------------------------------------- clocks

class Clocks:
    """nvidia-smi samples every 50 ms; summary() keeps those taken inside the
    window marked by start() / stop() (the timed region)."""
    Q = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.t0 = self.t1 = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        return self

    def start(self):
        import datetime
        self.t0 = datetime.datetime.now()

    def stop(self):
        import datetime
        self.t1 = datetime.datetime.now()

    def __exit__(self, *a):
        self.lines = []
        if self.proc:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        import datetime
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for l in getattr(self, "lines", []):
            f = [x.strip() for x in l.split(",")]
            if len(f) < 9:
                continue
            try:
                ts = datetime.datetime.strptime(f[0], "%Y/%m/%d %H:%M:%S.%f")
            except ValueError:
                ts = None  # unknown format: keep the sample
            if ts and self.t0 and self.t1 and not (self.t0 <= ts <= self.t1):
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------- set-up

def device_layer_weights(m, l, dev, gen, torch):
    qkv = (m.n_heads + 2 * m.n_kv_heads) * m.head_dim

    def rnd(shape):
        return (torch.randn(shape, device=dev, generator=gen, dtype=torch.float32) * 0.02).to(torch.bfloat16)

    return {"Wqkv": rnd((qkv, m.d)), "Wo": rnd((m.d, m.n_heads * m.head_dim)), "Wgu": rnd((2 * m.ffn, m.d)),
            "Wdown": rnd((m.d, m.ffn)), "attn_norm": torch.ones(m.d, device=dev),
            "mlp_norm": torch.ones(m.d, device=dev)}


def gemm_flops(w, T, K_sum, T_enc, n_txt_sum):
    """Algorithmic flops of every dense contraction of one step (2 per MAC)."""
    s, m = w.selector, w.model
    enc = s.n_enc_layers * 2.0 * T_enc * (3 * s.D * s.D + s.D * s.D + 2 * s.D * s.enc_ffn)
    text = 2.0 * n_txt_sum * s.D_text * s.D
    proj = 2.0 * K_sum * (m.proj_in * m.proj_hidden + m.proj_hidden * m.d) if m.proj_kind == "mlp2" else \
        (2.0 * K_sum * m.proj_in * m.d if m.proj_kind == "linear" else 0.0)
    qkv = (m.n_heads + 2 * m.n_kv_heads) * m.head_dim
    lm = m.n_layers * 2.0 * T * (m.d * qkv + m.n_heads * m.head_dim * m.d + 2 * m.d * m.ffn + m.ffn * m.d)
    return enc + text + proj + lm


_SAMPLE_CACHE = {}


def cpu_oracle_sample(w, n_images=1, n_layers=1):
    """Times the oracle on a bounded sample of the workload and scales it to one
    batch: per image the encoder + selection, the projector on its kept rows and
    n_layers of the 32 decoder layers (weights are drawn once, outside the timing)."""
    from oracle import core as O
    s, m = w.selector, w.model
    key = (w.name, n_layers)
    if key not in _SAMPLE_CACHE:
        _SAMPLE_CACHE[key] = (S.make_selector_weights(w), S.make_model_head(w), S.make_inputs(w),
                              [S.make_layer_weights(w, l) for l in range(n_layers)])
    sel, head, inp, layers = _SAMPLE_CACHE[key]
    n_heads = s.D // s.enc_head_dim
    t_sel = t_proj = t_lm = 0.0
    for b in range(n_images):
        v0, t0 = b * w.n_vis[0], b * w.n_txt[0]
        X = inp["X"][v0:v0 + w.n_vis[b]]
        E = inp["E_text"][t0:t0 + w.n_txt[b]]
        t = time.perf_counter()
        Et = O.text_projection(E, sel, s.ln_eps, s.g_text)
        H = O.encoder(X, Et, sel, n_heads, s.ln_eps)
        r = O.select_episode(H, sel, k_max=w.k_max, g=w.g, stop_bias=0.0, eps=s.ln_eps)
        idx = O.restore(r["order"])
        if len(idx) < int(w.target_mean_k):  # time a mean-sized prefix whatever this bias kept
            idx = np.arange(int(w.target_mean_k))
        t_sel += time.perf_counter() - t
        t = time.perf_counter()
        vis = O.projector(X[idx], head)
        t_proj += time.perf_counter() - t
        x = np.concatenate([vis, E])
        cu, pos = np.array([0, len(x)]), np.arange(len(x))
        t = time.perf_counter()
        for L in layers:
            x = O.prefill_layer(x, L, m, cu, pos)
        t_lm += time.perf_counter() - t
    per_image_ms = 1e3 * (t_sel + t_proj + t_lm * m.n_layers / n_layers) / n_images
    return per_image_ms * w.B, t_sel + t_proj + t_lm


def selection_report(B, w, selector, X, E, bias, kernel_ms, dev):
    """The selection kernel against its on-chip roofline: algorithmic bytes per
    round per episode are the folded pointer keys of its candidates, (N_e + 1) h
    fp32 from shared memory, the history rows the round's attention reads, 2 t h
    fp32 (t = history length) from the TMEM cache, and from L2 the rows that
    enter the round (the last position's query and residual rows, the key and
    value rows of the positions appended); the kernel's time is the longest
    episode's rounds.  Peaks and the synchronisation floor come from the
    library's probes."""
    r = B.sp_select(selector, w.n_vis, w.n_txt, X=X, E_text=E, stop_bias=bias, group_size=w.group_size, g=w.g,
                    k_max=w.k_max)
    import torch
    torch.cuda.synchronize()
    rounds = r["rounds"].cpu().numpy().astype(int)
    h = w.selector.h
    eps = w.episodes()
    n_max = max(n for (_, _, n) in eps)
    C = 8 if (n_max + 7) // 8 + 1 <= 128 else 16
    cached = C * 256 // (h // 128)  # history positions the TMEM cache of an episode holds
    smem_b = tmem_b = l2_b = 0.0
    for (_, _, n_e), R in zip(eps, rounds):
        for t_round in range(int(R)):
            t = min(1 + w.g * t_round, w.k_max)
            t_new = 1 if t_round == 0 else min(w.g, t - 1)
            smem_b += (n_e + 1) * h * 4.0
            in_tmem = max(0, min(t, cached) - t_new)
            tmem_b += 2.0 * in_tmem * h * 4.0
            l2_b += 2.0 * (t - in_tmem) * h * 4.0 + 2.0 * h * 4.0
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    smem_peak = B.probe_smem_gbs()
    l2_peak = B.probe_l2_gbs()
    r_max = int(rounds.max())
    floor_us = B.probe_select_floor(C, h, max(r_max, 1), len(eps))
    ks = kernel_ms * 1e-3
    used = min(len(eps) * C, sms) / sms
    onchip = smem_b + tmem_b + l2_b
    return {"kernel_ms": kernel_ms, "episodes": len(eps), "cluster_size": C, "max_rounds": r_max,
            "us_per_round": kernel_ms * 1e3 / max(r_max, 1), "floor_us_per_round": floor_us,
            "smem_bytes": smem_b, "tmem_bytes": tmem_b, "l2_bytes": l2_b,
            "smem_gbs": smem_b / ks / 1e9, "tmem_gbs": tmem_b / ks / 1e9, "l2_gbs": l2_b / ks / 1e9,
            "onchip_gbs": onchip / ks / 1e9,
            "smem_peak_gbs": smem_peak, "smem_peak_used_sms_gbs": smem_peak * used, "l2_peak_gbs": l2_peak,
            "onchip_frac_of_smem_peak_used_sms": onchip / ks / 1e9 / (smem_peak * used),
            "l2_frac": l2_b / ks / 1e9 / l2_peak,
            "note": "latency-bound dependent chain: compare us_per_round with floor_us_per_round"}


def cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    w = S.llava15_7b_b16()
    samples = []
    wall = 0.0
    for i in range(args.warmup + args.steps):
        v, secs = cpu_oracle_sample(w)
        wall += secs
        if i >= args.warmup:
            samples.append(v)
    value = statistics.median(samples)
    sample = ("per step: 1 of 16 images through text projection + 2-block encoder + selection, projector on "
              "its kept rows, 1 of 32 decoder layers; scaled to 16 images x 32 layers")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": value, "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": w.name, "images": w.B, "visual_tokens": w.n_vis[0], "text_tokens": w.n_txt[0],
                       "layers": w.model.n_layers},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores(), "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- our arm

def run_ours(args):
    import torch
    from paper_2609_13804_gb300 import binding as B

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")

    def barrier():
        if dist:
            dist.barrier()
        torch.cuda.synchronize()

    w = S.llava15_7b_b16(seed=1002 + rank)
    s, m = w.selector, w.model
    sel_w = S.make_selector_weights(w)
    selector = B.Selector(s, sel_w, dev)
    gen = torch.Generator(device=dev)
    gen.manual_seed(w.seed)
    layers = [device_layer_weights(m, l, dev, gen, torch) for l in range(m.n_layers)]
    head = {"final_norm": torch.ones(m.d, device=dev),
            "proj_W1": (torch.randn((m.proj_hidden, m.proj_in), device=dev, generator=gen) * 0.02).to(torch.bfloat16),
            "proj_W2": (torch.randn((m.d, m.proj_hidden), device=dev, generator=gen) * 0.02).to(torch.bfloat16)}
    model = B.Model(m, layers, head, dev, max_pos=1024)
    inp = S.make_inputs(w)
    X = B.dev_bf16(inp["X"], dev)
    E = B.dev_bf16(inp["E_text"], dev)
    n_ep = len(w.episodes())

    # STOP biases: gap traces with STOP disabled, then the realisable counts
    # nearest the per-image targets (16..192, mean 64)
    cal = B.sp_select(selector, w.n_vis, w.n_txt, X=X, E_text=E, stop_bias=B.dev_f32(np.full(n_ep, -1e30), dev),
                      group_size=w.group_size, g=w.g, k_max=w.k_max)
    torch.cuda.synchronize()
    gaps = cal["gap"].cpu().numpy()
    rounds = cal["rounds"].cpu().numpy()
    traces = [gaps[e, :rounds[e]] for e in range(n_ep)]
    biases, expect = S.stop_biases(traces, S.target_counts(w), g=w.g, k_max=w.k_max,
                                   n_cand=[n for (_, _, n) in w.episodes()], mean_target=w.target_mean_k)
    bias = B.dev_f32(biases, dev)

    pipe = B.Pipeline(selector, model, w.n_vis, w.n_txt, group_size=w.group_size, g=w.g, k_max=w.k_max)
    for _ in range(args.warmup):
        pipe(X, E, bias)
    torch.cuda.synchronize()
    if args.launch_list:
        # one more step and nothing else: the last step's launches are the list to read
        pipe(X, E, bias)
        torch.cuda.synchronize()
        return
    counts = pipe.count.cpu().numpy().astype(int)
    K_sum = int(counts.sum())
    T = int(pipe.cu[-1].item())
    T_enc = sum(w.n_vis) + sum(w.n_txt)
    flops = gemm_flops(w, T, K_sum, T_enc, sum(w.n_txt))

    # ---- timed region: K steps of the pipeline
    st = torch.cuda.current_stream()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with Clocks(local) as clk:
        time.sleep(0.3)  # let the sampler start; the warm GPU idles meanwhile
        pipe(X, E, bias)
        barrier()
        clk.start()
        ev0.record(st)
        for _ in range(args.steps):
            pipe(X, E, bias)
        ev1.record(st)
        barrier()
        clk.stop()
    ms_step = max_over_ranks(ev0.elapsed_time(ev1) / args.steps, dev)
    value = ms_step / world

    # ---- the same K steps again with CUDA events around every launch (on the
    #      launching stream): per-kernel-kind durations for the roofline; the
    #      events add host work per launch, so this pass is timed separately
    ev2, ev3 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    B.sp_profile_begin(args.steps * 2000)
    barrier()
    ev2.record(st)
    for _ in range(args.steps):
        pipe(X, E, bias)
    ev3.record(st)
    barrier()
    prof = B.sp_profile_end()
    ms_step_profiled = ev2.elapsed_time(ev3) / args.steps
    launches = sum(v["launches"] for v in prof.values()) // args.steps
    gemm_ms = prof["gemm"]["ms"] / args.steps
    pk = peaks()
    achieved = flops / (gemm_ms * 1e-3) / 1e12

    # ---- side measurements (outside the timed region)
    def timed(fn, reps=5):
        a, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        fn()
        torch.cuda.synchronize()
        a.record()
        for _ in range(reps):
            fn()
        b_.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b_) / reps

    sel_ws = None

    def do_select():
        nonlocal sel_ws
        r = B.sp_select(selector, w.n_vis, w.n_txt, X=X, E_text=E, stop_bias=bias, group_size=w.group_size,
                        g=w.g, k_max=w.k_max, traces=False, ws=sel_ws)
        sel_ws = r["_ws"]
        return r

    sel_out = do_select()
    select_ms = timed(do_select)
    k_cap = pipe.k_cap
    sel_report = selection_report(B, w, selector, X, E, bias, prof["select"]["ms"] / args.steps, dev)
    comp = {}

    def do_compact(idx, count, kc, reuse=False):
        prev = comp.get(kc) if reuse else None
        comp["o"] = comp[kc] = B.sp_compact(w.n_vis, w.n_txt, X=X, text=E, idx=idx, count=count, k_cap=kc,
                                            projector_mode=True, out=prev)

    def kernel_ms(fn, reps=5):
        # device time per call of a one-launch call: a spin kernel ahead of the
        # calls keeps the GPU busy while the host enqueues them, so they run
        # back to back between one pair of events (no host gap, no per-launch
        # events inside)
        fn()
        torch.cuda.synchronize()
        a, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda._sleep(4_000_000)
        a.record()
        for _ in range(reps):
            fn()
        b_.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b_) / reps

    flush_buf = torch.empty(256 << 20, dtype=torch.uint8, device=dev)  # twice the L2

    def kernel_ms_cold(fn, reps=10):
        # device time of a one-launch call with L2 flushed before each call (its
        # inputs are smaller than L2): flush, then a spin kernel so the host has
        # enqueued the events and the call before the GPU reaches them
        fn()
        total = 0.0
        for _ in range(reps):
            flush_buf.zero_()
            a, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda._sleep(1_000_000)
            a.record()
            fn()
            b_.record()
            torch.cuda.synchronize()
            total += a.elapsed_time(b_)
        return total / reps

    compact_ms = kernel_ms_cold(lambda: do_compact(sel_out["idx"], sel_out["count"], k_cap, reuse=True))
    comp_bytes = 2.0 * (K_sum * s.D + sum(w.n_txt) * m.d) * 2 + 4.0 * (w.B + 1 + T)

    def prefill_stage(idx, count, kc):
        do_compact(idx, count, kc)
        o = comp["o"]
        B.sp_project(model, vis_packed=o["vis_packed"], vis_row_map=o["vis_row_map"], vis_cu=o["vis_cu"],
                     packed=o["packed"], rows_cap=o["rows_cap"], B=w.B)
        lens_cap = max(min(n, kc) + t for n, t in zip(w.n_vis, w.n_txt))
        B.sp_prefill(model, x=o["packed"], cu_seqlens=o["cu_seqlens"], pos=o["pos"], B=w.B, T_cap=o["T_cap"],
                     max_seqlen_cap=lens_cap)

    pruned_ms = timed(lambda: prefill_stage(sel_out["idx"], sel_out["count"], k_cap), reps=3)
    full_idx = torch.arange(576, dtype=torch.int32, device=dev).repeat(w.B, 1).contiguous()
    full_cnt = torch.full((w.B,), 576, dtype=torch.int32, device=dev)
    full_ms = timed(lambda: prefill_stage(full_idx, full_cnt, 576), reps=3)
    # per-kind split of one full-prefix pass (events around every launch): the
    # attention at 624-token sequences, where it has enough work to be bound by
    # the tensor pipe rather than by launch latency
    B.sp_profile_begin(4000)
    prefill_stage(full_idx, full_cnt, 576)
    torch.cuda.synchronize()
    full_prof = B.sp_profile_end()
    full_lens = [n + t for n, t in zip(w.n_vis, w.n_txt)]
    attn_full_flops = 4.0 * m.n_heads * m.head_dim * sum(L * (L + 1) / 2 for L in full_lens) * m.n_layers
    attn_full_ms = full_prof["attention"]["ms"]
    # compaction at a bandwidth-sized case: every visual token kept (the full prefix)
    full_compact_ms = kernel_ms_cold(lambda: do_compact(full_idx, full_cnt, 576, reuse=True))
    full_T = sum(w.n_vis) + sum(w.n_txt)
    full_comp_bytes = 2.0 * (sum(w.n_vis) * s.D + sum(w.n_txt) * m.d) * 2 + 4.0 * (w.B + 1 + full_T)
    # bandwidth-sized compaction: 128 images, every visual token kept (201 MB
    # read + 201 MB written, above the L2's 126 MB), timed back to back
    nbig = 128
    Xbig = torch.randn((nbig * 576, s.D), device=dev, generator=gen).to(torch.bfloat16)
    Ebig = (torch.randn((nbig * 48, m.d), device=dev, generator=gen) * 0.02).to(torch.bfloat16)
    big_idx = torch.arange(576, dtype=torch.int32, device=dev).repeat(nbig, 1).contiguous()
    big_cnt = torch.full((nbig,), 576, dtype=torch.int32, device=dev)
    big_nv, big_nt = [576] * nbig, [48] * nbig
    big_out = B.sp_compact(big_nv, big_nt, X=Xbig, text=Ebig, idx=big_idx, count=big_cnt, k_cap=576,
                           projector_mode=True)
    big_ms = kernel_ms(lambda: B.sp_compact(big_nv, big_nt, X=Xbig, text=Ebig, idx=big_idx, count=big_cnt,
                                            k_cap=576, projector_mode=True, out=big_out), reps=10)
    big_bytes = 2.0 * (nbig * 576 * s.D + nbig * 48 * m.d) * 2 + 4.0 * (nbig + 1 + nbig * 624)
    del Xbig, Ebig, big_out

    # ---- generation over the pruned prefix vs the full prefix (one token per
    #      sequence per step, 32 layers; the cache contents do not change the
    #      work, so a zeroed cache with the prefix lengths stands in)
    def decode_ms(lens, steps=20, warm=3):
        S_cap = max(lens) + warm + steps + 8
        kv = B.kv_cache(model, w.B, S_cap)
        x_new = (torch.randn((w.B, m.d), device=dev, generator=gen) * 0.5).to(torch.bfloat16)
        lens_d = torch.tensor(lens, dtype=torch.int32, device=dev)
        o = B.sp_decode(model, x=x_new, lens=lens_d, kv=kv, max_len_cap=S_cap)
        ws_d = o["_ws"]
        for _ in range(warm - 1):
            B.sp_decode(model, x=x_new, lens=lens_d, kv=kv, max_len_cap=S_cap, ws=ws_d)
        lens_d.copy_(torch.tensor(lens, dtype=torch.int32, device=dev))
        torch.cuda.synchronize()
        a, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(steps):
            B.sp_decode(model, x=x_new, lens=lens_d, kv=kv, max_len_cap=S_cap, ws=ws_d)
        b_.record()
        torch.cuda.synchronize()
        del kv
        return a.elapsed_time(b_) / steps

    pruned_lens = np.diff(pipe.cu.cpu().numpy()).astype(int).tolist()
    full_lens = [n + t for n, t in zip(w.n_vis, w.n_txt)]
    dec_pruned_ms = decode_ms(pruned_lens)
    dec_full_ms = decode_ms(full_lens)
    qkv_w = (m.n_heads + 2 * m.n_kv_heads) * m.head_dim
    weight_bytes = 2.0 * m.n_layers * (m.d * qkv_w + m.n_heads * m.head_dim * m.d + 3 * m.d * m.ffn)

    def cache_bytes(lens):
        return 2.0 * 2 * m.n_layers * m.n_kv_heads * m.head_dim * sum(n + 1 for n in lens)

    # ---- the training-time pathway's forward on the same batch (Eqs. 5-9):
    #      the rollout with its aggregates (same STOP biases, so the same
    #      trajectory as the timed selection), SoftTopK, the gate on X
    def do_train_select():
        return B.sp_select(selector, w.n_vis, w.n_txt, X=X, E_text=E, stop_bias=bias, group_size=w.group_size,
                           g=1, k_max=w.k_max, traces=False, ws=sel_ws, train=(1.0, 0.99))

    tr = do_train_select()
    select_train_ms = timed(do_train_select)
    alpha_buf = torch.empty(sum(w.n_vis), dtype=torch.float32, device=dev)
    topk_ms = kernel_ms(lambda: B.sp_soft_topk(w.n_vis, score=tr["score"], kbar=tr["kbar"], tau=0.05,
                                               group_size=w.group_size, alpha=alpha_buf))
    noise = torch.randn(X.shape, device=dev, generator=gen).to(torch.bfloat16)
    gated = torch.empty_like(X)
    gate_ms = kernel_ms(lambda: B.sp_vp_gate(X=X, noise=noise, alpha=alpha_buf, out=gated))
    gate_bytes = 3.0 * X.numel() * 2
    del noise, gated
    # bandwidth-sized gate: 256 images of 576 tokens (0.9 GB moved)
    big_rows = 256 * 576
    Xg = torch.randn((big_rows, s.D), device=dev, generator=gen).to(torch.bfloat16)
    Ng = torch.randn((big_rows, s.D), device=dev, generator=gen).to(torch.bfloat16)
    Ag = torch.rand(big_rows, device=dev, generator=gen)
    Og = torch.empty_like(Xg)
    gate_big_ms = kernel_ms(lambda: B.sp_vp_gate(X=Xg, noise=Ng, alpha=Ag, out=Og))
    gate_big_bytes = 3.0 * Xg.numel() * 2
    del Xg, Ng, Ag, Og

    # ---- pointer decoders of one and of two layers on the same shapes (every
    #      episode runs its 192 rounds: STOP disabled; memory H given)
    Hm = B.dev_f32(S.make_memory(w), dev)
    nostop = B.dev_f32(np.full(w.B, -1e30), dev)
    deep = {}
    for nd in (1, 2):
        shp = dataclasses.replace(s, n_enc_layers=0, n_dec_layers=nd)
        dsel = B.Selector(shp, S.make_selector_weights(dataclasses.replace(w, selector=shp)), dev)
        dws = [None]

        def run_deep():
            r = B.sp_select(dsel, w.n_vis, w.n_txt, H=Hm, stop_bias=nostop, g=1, k_max=w.k_max, traces=False,
                            ws=dws[0])
            dws[0] = r["_ws"]

        deep[nd] = timed(run_deep)
        dsel.close()
    del Hm

    # ---- end to end from host buffers (copies inside the timed region)
    Xh = X.cpu().pin_memory()
    Eh = E.cpu().pin_memory()
    bh = bias.cpu().pin_memory()
    oi = torch.empty(pipe.idx.shape, dtype=torch.int32).pin_memory()
    oc = torch.empty(pipe.count.shape, dtype=torch.int32).pin_memory()
    ocu = torch.empty(pipe.cu.shape, dtype=torch.int32).pin_memory()
    oh = torch.empty(pipe.hidden.shape, dtype=torch.float32).pin_memory()
    pipe.host(Xh, Eh, bh, oi, oc, ocu, oh)
    torch.cuda.synchronize()
    e2e_steps = max(2, min(args.steps, 5))
    barrier()
    a, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(e2e_steps):
        pipe.host(Xh, Eh, bh, oi, oc, ocu, oh)
    b_.record()
    barrier()
    e2e_ms = max_over_ranks(a.elapsed_time(b_) / e2e_steps, dev)
    h2d = Xh.numel() * 2 + Eh.numel() * 2 + bh.numel() * 4
    d2h = oi.numel() * 4 + oc.numel() * 4 + ocu.numel() * 4 + oh.numel() * 4

    if rank == 0:
        cpu_line = None
        if world == 1 and not args.no_cpu:
            v, secs = cpu_oracle_sample(w)
            cpu_line = {"value": v, "unit": UNIT, "cores": cores(), "kind": "oracle",
                        "sample": "1 of 16 images (encoder + selection, projector, 1 of 32 layers), scaled to "
                                  f"16 images x 32 layers; {secs:.1f} s of CPU work"}
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": False, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": w.name, "images": w.B, "visual_tokens": w.n_vis[0], "text_tokens": w.n_txt[0],
                       "layers": m.n_layers, "d": m.d, "selector_h": s.h, "k_max": w.k_max,
                       "mean_kept": float(counts.mean()), "packed_tokens": T,
                       "l2": "inputs larger than L2: 13.5 GB of weights streamed every step"},
            "roofline": {"kernel": "gemm_tc (tcgen05)", "bound": "tensor", "achieved": achieved,
                         "peak": pk["bf16_sus"], "unit": "TFLOP/s", "frac": achieved / pk["bf16_sus"],
                         "peak_source": pk["source"] + " bf16 sustained", "traffic": gemm_traffic(),
                         "traffic_unit": "DRAM bytes per launch",
                         "gemm_ms_per_step": gemm_ms, "gemm_flops_per_step": flops},
            "cpu_baseline": cpu_line,
            "e2e": {"value": e2e_ms / world, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
            "gpu_launches": launches,
            "clocks": clk.summary(),
            "stages_ms_per_step": {k: v["ms"] / args.steps for k, v in prof.items()},
            "ms_per_step_with_launch_events": ms_step_profiled,
            "select_us_per_image": 1e3 * select_ms / w.B,
            "selection": sel_report,
            "compaction_gbs": comp_bytes / (compact_ms * 1e-3) / 1e9,
            "compaction_full_prefix_gbs": full_comp_bytes / (full_compact_ms * 1e-3) / 1e9,
            "compaction_full_prefix_hbm_frac": full_comp_bytes / (full_compact_ms * 1e-3) / 1e9 / pk["hbm_gbs"],
            "compaction_128_images_gbs": big_bytes / (big_ms * 1e-3) / 1e9,
            "compaction_128_images_hbm_frac": big_bytes / (big_ms * 1e-3) / 1e9 / pk["hbm_gbs"],
            "compaction_note": ("16-image figures: one call after an L2 flush, events around it (launch latency "
                                "included); 128 images: 402 MB moved per call, back to back"),
            "attention_full_prefix": {
                "ms": attn_full_ms, "layers": m.n_layers, "sequences": w.B, "seq_len": full_lens[0],
                "algorithmic_tflops": attn_full_flops / (attn_full_ms * 1e-3) / 1e12,
                "frac_of_bf16_burst": attn_full_flops / (attn_full_ms * 1e-3) / 1e12 / pk["bf16"],
                "note": "causal flops 4 H d_h sum L(L+1)/2 per layer; events around each launch"},
            "pruned_prefill_ms": pruned_ms,
            "full_prefix_prefill_ms": full_ms,
            "speedup_prefill": full_ms / pruned_ms,
            "speedup_with_selection": full_ms / (pruned_ms + select_ms),
            "token_ratio": (sum(w.n_vis) + sum(w.n_txt)) / T,
            "kept_counts": counts.tolist(),
            "decode": {"ms_per_step_pruned_prefix": dec_pruned_ms, "ms_per_step_full_prefix": dec_full_ms,
                       "speedup": dec_full_ms / dec_pruned_ms, "sequences": w.B,
                       "hbm_gbs_pruned": (weight_bytes + cache_bytes(pruned_lens)) / (dec_pruned_ms * 1e-3) / 1e9,
                       "hbm_frac_pruned": (weight_bytes + cache_bytes(pruned_lens)) / (dec_pruned_ms * 1e-3) / 1e9
                       / pk["hbm_gbs"],
                       "bytes_note": "weights of the 32 layers + the cache rows read, per step"},
            "train_forward": {
                "select_ms": select_ms, "select_train_ms": select_train_ms,
                "aggregates_overhead": select_train_ms / select_ms - 1.0,
                "soft_topk_us": 1e3 * topk_ms, "vp_gate_us": 1e3 * gate_ms,
                "vp_gate_gbs": gate_bytes / (gate_ms * 1e-3) / 1e9,
                "vp_gate_256_images_gbs": gate_big_bytes / (gate_big_ms * 1e-3) / 1e9,
                "vp_gate_256_images_hbm_frac": gate_big_bytes / (gate_big_ms * 1e-3) / 1e9 / pk["hbm_gbs"],
                "note": "tau 1.0, beta 0.99, SoftTopK tau 0.05; the gate reads X and noise, writes the gated rows"},
            "deep_decoder": {
                "select_1_layer_ms": deep[1], "select_2_layers_ms": deep[2], "rounds": w.k_max,
                "us_per_round_1_layer": 1e3 * deep[1] / w.k_max, "us_per_round_2_layers": 1e3 * deep[2] / w.k_max,
                "note": "16 episodes x 192 rounds from a given memory H (precompute GEMMs included)"},
        }
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


# Sec. 4 scaling table (LLaVA-1.5-7B rows): input tokens, retained tokens,
# full prefill ms, pruned-path ms, selector ms, on the paper's GPU (context only)
PAPER_SCALING = {
    320: (32, 29.34, 30.00, 9.65), 640: (64, 53.24, 37.14, 16.15), 960: (96, 70.86, 37.75, 20.45),
    1280: (128, 116.89, 40.91, 24.25), 1600: (160, 142.93, 46.13, 28.85), 1920: (192, 189.83, 52.28, 34.41),
    2240: (224, 236.55, 57.73, 39.14)}


def run_sweep(args):
    """Scaling with the visual-prefix length at 10% retention: one image of N
    visual + 48 text tokens on the LLaVA-1.5-7B-shaped model, N = 320..2240.
    Per N: the full-prefix prefill (projector on N rows + 32 layers over N + 48),
    the pruned path (selector incl. its encoder, compaction, projector on the
    kept rows, 32 layers over K + 48) and the selector alone, each the mean of
    `--steps` calls after `--warmup`."""
    import torch
    from paper_2609_13804_gb300 import binding as B

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    w = S.llava15_7b_b16()
    s, m = w.selector, w.model
    selector = B.Selector(s, S.make_selector_weights(w), dev)
    gen = torch.Generator(device=dev)
    gen.manual_seed(w.seed)
    layers = [device_layer_weights(m, l, dev, gen, torch) for l in range(m.n_layers)]
    head = {"final_norm": torch.ones(m.d, device=dev),
            "proj_W1": (torch.randn((m.proj_hidden, m.proj_in), device=dev, generator=gen) * 0.02).to(torch.bfloat16),
            "proj_W2": (torch.randn((m.d, m.proj_hidden), device=dev, generator=gen) * 0.02).to(torch.bfloat16)}
    model = B.Model(m, layers, head, dev, max_pos=4096)
    L = 48

    def timed(fn):
        for _ in range(args.warmup):
            fn()
        torch.cuda.synchronize()
        a, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(args.steps):
            fn()
        b_.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b_) / args.steps

    rows = []
    for N in sorted(PAPER_SCALING):
        K = N // 10
        X = (torch.randn((N, s.D), device=dev, generator=gen)).to(torch.bfloat16)
        E = (torch.randn((L, m.d), device=dev, generator=gen) * 0.02).to(torch.bfloat16)
        bias = torch.full((1,), -1e30, dtype=torch.float32, device=dev)  # STOP never wins: exactly K kept
        pipe = B.Pipeline(selector, model, [N], [L], group_size=0, g=1, k_max=K)
        pruned_ms = timed(lambda: pipe(X, E, bias))
        sel_ws = {}

        def select():
            r = B.sp_select(selector, [N], [L], X=X, E_text=E, stop_bias=bias, group_size=0, g=1, k_max=K,
                            traces=False, ws=sel_ws.get("ws"))
            sel_ws["ws"] = r["_ws"]
        selector_ms = timed(select)
        full_idx = torch.arange(N, dtype=torch.int32, device=dev).reshape(1, N)
        full_cnt = torch.full((1,), N, dtype=torch.int32, device=dev)
        st = {}

        def full_prefill():
            o = B.sp_compact([N], [L], X=X, text=E, idx=full_idx, count=full_cnt, k_cap=N, projector_mode=True,
                             out=st.get("c"))
            st["c"] = o
            B.sp_project(model, vis_packed=o["vis_packed"], vis_row_map=o["vis_row_map"], vis_cu=o["vis_cu"],
                         packed=o["packed"], rows_cap=o["rows_cap"], B=1)
            r = B.sp_prefill(model, x=o["packed"], cu_seqlens=o["cu_seqlens"], pos=o["pos"], B=1, T_cap=o["T_cap"],
                             max_seqlen_cap=N + L, ws=st.get("ws"), hidden=st.get("h"))
            st["ws"], st["h"] = r["_ws"], r["hidden"]
        full_ms = timed(full_prefill)
        kept = int(pipe.count[0].item())
        pk, pf, pp, ps = PAPER_SCALING[N]
        rows.append({"input_tokens": N, "retained": kept, "full_prefill_ms": full_ms, "stepprune_prefill_ms": pruned_ms,
                     "selector_ms": selector_ms, "speedup": full_ms / pruned_ms,
                     "selector_share": selector_ms / pruned_ms,
                     "paper": {"retained": pk, "full_prefill_ms": pf, "stepprune_prefill_ms": pp, "selector_ms": ps,
                               "speedup": pf / pp, "selector_share": ps / pp}})
        del pipe
    line = {"sweep": "visual-prefix length at 10% retention", "config": {"workload": "llava15-7b dims, 1 image",
            "text_tokens": L, "layers": m.n_layers}, "steps": args.steps, "warmup": args.warmup,
            "paper_gpu": "RTX PRO 6000 Blackwell (the paper's; context only)", "rows": rows}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu", action="store_true", help="skip the CPU oracle baseline")
    ap.add_argument("--launch-list", action="store_true",
                    help="set up, warm up and run one more step only (for an ncu launch list)")
    ap.add_argument("--sweep", action="store_true",
                    help="scaling with the visual-prefix length at 10%% retention (one JSON line, no headline)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.sweep:
        run_sweep(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
