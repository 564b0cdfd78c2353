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
GEMM_TRAFFIC = {"bytes_per_launch": 163.7e6, "sources_sha256_16": "87fbbb39393a6906"}
GEMM_SOURCES = ("paper_2609_13804_gb300/csrc/gemm_tc.cu", "paper_2609_13804_gb300/csrc/common.cuh")


# DRAM read + write bytes of one full-prefix attention launch (16 x 624 tokens,
# 32 heads of 128, causal; the head-pair kernel) from the ncu capture summarised
# in profiles/attn_pair_kernel_llava15-7b-dims_full_prefix.md, valid for the
# kernel sources with this digest.
ATTN_TRAFFIC = {"bytes_per_launch": 322.0e6, "sources_sha256_16": "544923811917fe9d"}
ATTN_SOURCES = ("paper_2609_13804_gb300/csrc/attention.cu", "paper_2609_13804_gb300/csrc/common.cuh")


def _digest(paths):
    import hashlib
    h = hashlib.sha256()
    for rel in paths:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def gemm_traffic():
    return GEMM_TRAFFIC["bytes_per_launch"] if _digest(GEMM_SOURCES) == GEMM_TRAFFIC["sources_sha256_16"] else None


def attn_traffic():
    return ATTN_TRAFFIC["bytes_per_launch"] if _digest(ATTN_SOURCES) == ATTN_TRAFFIC["sources_sha256_16"] else None


PROBES_SRC = os.path.join(ROOT, "bench_probes.cu")
PROBES_LIB = os.path.join(ROOT, "bench_probes.so")


def build_probes() -> str:
    """Compiles bench_probes.cu (the on-chip peak and synchronisation-floor
    probes this script reports against) for sm_103a, next to this file."""
    if os.path.exists(PROBES_LIB) and os.path.getmtime(PROBES_LIB) >= os.path.getmtime(PROBES_SRC):
        return PROBES_LIB
    from paper_2609_13804_gb300.build import _nvcc, ARCH
    tmp = PROBES_LIB + ".tmp"
    subprocess.run([_nvcc(), *ARCH, "-O3", "-std=c++17", "-shared", "-Xcompiler", "-fPIC", PROBES_SRC, "-o", tmp],
                   check=True, capture_output=True, text=True)
    os.replace(tmp, PROBES_LIB)
    return PROBES_LIB


class Probes:
    """ctypes view of bench_probes.so."""

    def __init__(self):
        import ctypes as C
        self.C = C
        self.lib = C.CDLL(build_probes())
        for n in ("bench_probe_smem_gbs", "bench_probe_l2_gbs"):
            getattr(self.lib, n).argtypes = [C.POINTER(C.c_double)]
            getattr(self.lib, n).restype = C.c_int
        self.lib.bench_probe_select_floor.argtypes = [C.c_int, C.c_int, C.c_int, C.c_int, C.POINTER(C.c_double)]
        self.lib.bench_probe_select_floor.restype = C.c_int

    def _call(self, fn, *args):
        v = self.C.c_double()
        rc = fn(*args, self.C.byref(v))
        if rc != 0:
            raise RuntimeError(f"{fn.__name__}: CUDA error {rc}")
        return v.value

    def smem_gbs(self):
        return self._call(self.lib.bench_probe_smem_gbs)

    def l2_gbs(self):
        return self._call(self.lib.bench_probe_l2_gbs)

    def select_floor(self, cluster_size, h, rounds, episodes):
        return self._call(self.lib.bench_probe_select_floor, cluster_size, h, rounds, episodes)


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


def cpu_oracle_sample(w, b=0, n_layers=1):
    """Times the oracle on a bounded sample of the workload: image b through
    the text projection, the encoder and the selection with that image's
    calibrated STOP bias (the GPU's kept-count target for it), the projector on
    its kept rows, and n_layers of the 32 decoder layers over its packed
    sequence.  Weights are drawn and the bias calibrated once, outside the
    timing.  Returns (the batch time extrapolated from the sample in ms, the
    measured parts in seconds)."""
    from oracle import core as O
    s, m = w.selector, w.model
    key = (w.name, n_layers)
    if key not in _SAMPLE_CACHE:
        _SAMPLE_CACHE[key] = (S.make_selector_weights(w), S.make_model_head(w), S.make_inputs(w),
                              [S.make_layer_weights(w, l) for l in range(n_layers)], {})
    sel, head, inp, layers, biases = _SAMPLE_CACHE[key]
    n_heads = s.D // s.enc_head_dim
    v0, t0 = sum(w.n_vis[:b]), sum(w.n_txt[:b])
    X = inp["X"][v0:v0 + w.n_vis[b]]
    E = inp["E_text"][t0:t0 + w.n_txt[b]]
    if b not in biases:
        Et = O.text_projection(E, sel, s.ln_eps, s.g_text)
        H = O.encoder(X, Et, sel, n_heads, s.ln_eps)
        free = O.select_episode(H, sel, k_max=w.k_max, g=w.g, stop_bias=-1e30, eps=s.ln_eps)
        bias, _ = S.stop_biases([free["gap"]], [int(S.target_counts(w)[b])], g=w.g, k_max=w.k_max,
                                n_cand=[w.n_vis[b]])
        biases[b] = float(bias[0])
    t = time.perf_counter()
    Et = O.text_projection(E, sel, s.ln_eps, s.g_text)
    H = O.encoder(X, Et, sel, n_heads, s.ln_eps)
    r = O.select_episode(H, sel, k_max=w.k_max, g=w.g, stop_bias=biases[b], eps=s.ln_eps)
    idx = O.restore(r["order"])
    t_sel = time.perf_counter() - t
    t = time.perf_counter()
    vis = O.projector(X[idx], head)
    t_proj = time.perf_counter() - t
    x = np.concatenate([vis, E])
    cu, pos = np.array([0, len(x)]), np.arange(len(x))
    t = time.perf_counter()
    for L in layers:
        x = O.prefill_layer(x, L, m, cu, pos)
    t_lm = (time.perf_counter() - t) / n_layers
    per_image_ms = 1e3 * (t_sel + t_proj + t_lm * m.n_layers)
    return per_image_ms * w.B, {"select_s": t_sel, "projector_s": t_proj, "layer_s": t_lm, "kept": int(len(idx)),
                                "image": b}


def selection_report(B, w, selector, X, E, bias, kernel_ms, dev):
    """The selection kernel against its on-chip roofline: algorithmic bytes per
    round per episode are the folded pointer keys of its candidates, (N_e + 1) h
    fp32 from shared memory, the history rows the round's attention reads, 2 t h
    fp32 (t = history length) from the TMEM cache, and from L2 the rows that
    enter the round (the last position's query and residual rows, the key and
    value rows of the positions appended); the kernel's time is the longest
    episode's rounds.  Peaks and the synchronisation floor come from the
    probes of bench_probes.cu."""
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
    probes = Probes()
    smem_peak = probes.smem_gbs()
    l2_peak = probes.l2_gbs()
    r_max = int(rounds.max())
    floor_us = probes.select_floor(C, h, max(r_max, 1), len(eps))
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


def run_reference(args, w=None):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    w = w or S.llava15_7b_b16()
    samples, parts = [], []
    for i in range(args.warmup + args.steps):
        v, part = cpu_oracle_sample(w, b=i % w.B)
        if i >= args.warmup:
            samples.append(v)
            parts.append(part)
    value = statistics.median(samples)
    sample = ("per step: one of the 16 images (in turn) through text projection + 2-block encoder + selection with "
              "its calibrated STOP bias, the projector on its kept rows and 1 of the 32 decoder layers over its "
              "packed sequence; extrapolated to 16 images x 32 layers")
    measured = {"select_s_median": statistics.median(p["select_s"] for p in parts),
                "projector_s_median": statistics.median(p["projector_s"] for p in parts),
                "layer_s_median": statistics.median(p["layer_s"] for p in parts),
                "kept": [p["kept"] for p in parts]}
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": value, "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": w.name, "images": w.B, "visual_tokens": w.n_vis[0], "text_tokens": w.n_txt[0],
                       "layers": w.model.n_layers},
            "extrapolated": True, "samples_timed": len(samples), "measured": measured,
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores(), "kind": "oracle", "sample": sample,
                             "extrapolated": True,
                             "threads": "numpy's BLAS may spread a matmul over the cores; the selection and "
                                        "attention loops run on one"},
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

    # the global batch holds `world` replicas' worth of images (weak scaling),
    # drawn once from one seed; each rank takes its share of the images
    # (longest-first greedy on the token counts: replicas.shard_images) and
    # runs it on an identical copy of the weights
    from paper_2609_13804_gb300.replicas import shard_images
    w1 = S.llava15_7b_b16()
    wg = dataclasses.replace(w1, n_vis=list(w1.n_vis) * world, n_txt=list(w1.n_txt) * world)
    mine = shard_images(wg.n_vis, wg.n_txt, world, rank)
    w = dataclasses.replace(w1, n_vis=[wg.n_vis[b] for b in mine], n_txt=[wg.n_txt[b] for b in mine])
    s, m = w.selector, w.model
    sel_w = S.make_selector_weights(w)
    selector = B.Selector(s, sel_w, dev)
    gen = torch.Generator(device=dev)
    gen.manual_seed(w.seed)
    layers = [device_layer_weights(m, l, dev, gen, torch) for l in range(m.n_layers)]
    head = {"final_norm": torch.ones(m.d, device=dev),
            "proj_W1": (torch.randn((m.proj_hidden, m.proj_in), device=dev, generator=gen) * 0.02).to(torch.bfloat16),
            "proj_W2": (torch.randn((m.d, m.proj_hidden), device=dev, generator=gen) * 0.02).to(torch.bfloat16)}
    model = B.Model(m, layers, head, dev, max_pos=4096)
    inp_g = S.make_inputs(wg)
    ov, ot = np.cumsum([0] + list(wg.n_vis)), np.cumsum([0] + list(wg.n_txt))
    inp = {"X": np.concatenate([inp_g["X"][ov[b]:ov[b + 1]] for b in mine]),
           "E_text": np.concatenate([inp_g["E_text"][ot[b]:ot[b + 1]] for b in mine])}
    del inp_g
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

    # ---- the per-step distribution: max(K, 20) more steps, an event pair around
    #      each (async records, no synchronisation between steps)
    n_dist = max(args.steps, 20)
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(n_dist + 1)]
    barrier()
    evs[0].record(st)
    for i in range(n_dist):
        pipe(X, E, bias)
        evs[i + 1].record(st)
    torch.cuda.synchronize()
    per_step = sorted(evs[i].elapsed_time(evs[i + 1]) for i in range(n_dist))
    pct = lambda q: per_step[min(n_dist - 1, int(round(q * (n_dist - 1))))]
    step_dist = {"steps": n_dist, "p10_ms": pct(0.1), "median_ms": pct(0.5), "p90_ms": pct(0.9),
                 "min_ms": per_step[0], "max_ms": per_step[-1]}

    # ---- the same step captured once in a CUDA graph and replayed K times
    #      (the call is capture-safe); reported beside the value
    graph_ms = None
    try:
        gph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gph):
            pipe(X, E, bias)
        gph.replay()
        barrier()
        ev4, ev5 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ev4.record(st)
        for _ in range(args.steps):
            gph.replay()
        ev5.record(st)
        barrier()
        graph_ms = max_over_ranks(ev4.elapsed_time(ev5) / args.steps, dev)
        del gph
    except Exception as ex:  # (a capture the runtime refuses: reported, not fatal)
        print(f"pipeline graph capture: {ex}", file=sys.stderr)

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

    icomp = {}

    def prefill_stage(idx, count, kc):
        # the pipeline's form: index-mode compaction, the projector gathering the kept rows of X
        o = icomp[kc] = B.sp_compact(w.n_vis, w.n_txt, X=X, text=E, idx=idx, count=count, k_cap=kc,
                                     index_mode=True, out=icomp.get(kc))
        B.sp_project(model, X=X, vis_src=o["vis_src"], vis_row_map=o["vis_row_map"], vis_cu=o["vis_cu"],
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
    def decode_ms(lens, steps=20, warm=3, graph=False):
        """ms per generation step: each step issued through sp_decode, or (graph)
        one step captured in a CUDA graph and replayed (the step is
        capture-safe: the lengths live and advance on the device)."""
        S_cap = max(lens) + warm + 2 * steps + 8
        kv = B.kv_cache(model, w.B, S_cap)
        x_new = (torch.randn((w.B, m.d), device=dev, generator=gen) * 0.5).to(torch.bfloat16)
        hid = torch.zeros((w.B, m.d), dtype=torch.float32, device=dev)
        lens_d = torch.tensor(lens, dtype=torch.int32, device=dev)
        o = B.sp_decode(model, x=x_new, lens=lens_d, kv=kv, max_len_cap=S_cap, hidden=hid)
        ws_d = o["_ws"]
        for _ in range(warm - 1):
            B.sp_decode(model, x=x_new, lens=lens_d, kv=kv, max_len_cap=S_cap, ws=ws_d, hidden=hid)
        step = lambda: B.sp_decode(model, x=x_new, lens=lens_d, kv=kv, max_len_cap=S_cap, ws=ws_d, hidden=hid)
        if graph:
            g = torch.cuda.CUDAGraph()
            torch.cuda.synchronize()
            with torch.cuda.graph(g):
                step()
            step = g.replay
        lens_d.copy_(torch.tensor(lens, dtype=torch.int32, device=dev))
        torch.cuda.synchronize()
        a, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(steps):
            step()
        b_.record()
        torch.cuda.synchronize()
        del kv
        return a.elapsed_time(b_) / steps

    pruned_lens = np.diff(pipe.cu.cpu().numpy()).astype(int).tolist()
    full_lens = [n + t for n, t in zip(w.n_vis, w.n_txt)]
    dec_pruned_ms = decode_ms(pruned_lens)
    dec_full_ms = decode_ms(full_lens)
    try:
        dec_graph_ms = decode_ms(pruned_lens, graph=True)
    except Exception as ex:  # (a capture the runtime refuses: reported, not fatal)
        print(f"decode graph capture: {ex}", file=sys.stderr)
        dec_graph_ms = None
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

    # ---- the other workloads (their own weights and inputs, drawn on the
    #      device) and the scaling table, outside the timed region
    workloads = scaling = None
    if not args.no_configs:
        workloads = measure_workloads(B, torch, dev, gen, peaks(), model)
        scaling = {"sweep": "visual-prefix length at 10% retention, one image, llava15-7b dims, 32 layers",
                   "steps": 3, "warmup": 1, "paper_gpu": "RTX PRO 6000 Blackwell (the paper's; context only)",
                   "rows": scaling_rows(B, torch, dev, gen, selector, model, 3, 1)}

    if rank == 0:
        cpu_line = None
        if world == 1 and not args.no_cpu:
            v, part = cpu_oracle_sample(w)
            cpu_line = {"value": v, "unit": UNIT, "cores": cores(), "kind": "oracle", "extrapolated": True,
                        "measured": part,
                        "threads": "numpy's BLAS may spread a matmul over the cores; the selection and attention "
                                   "loops run on one",
                        "sample": "image 0 (encoder + selection with its calibrated STOP bias, projector on its "
                                  "kept rows, 1 of 32 layers), extrapolated to 16 images x 32 layers"}
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": False, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": w.name, "images": w.B, "global_images": wg.B,
                       "sharding": "each rank its share of one global batch (replicas.shard_images); no collective",
                       "visual_tokens": w.n_vis[0], "text_tokens": w.n_txt[0],
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
            "step_distribution": step_dist,
            "ms_per_step_cuda_graph": graph_ms,
            "select_us_per_image": 1e3 * select_ms / w.B,
            "selection": sel_report,
            "compaction_gbs": comp_bytes / (compact_ms * 1e-3) / 1e9,
            "compaction_full_prefix_gbs": full_comp_bytes / (full_compact_ms * 1e-3) / 1e9,
            "compaction_full_prefix_hbm_frac": full_comp_bytes / (full_compact_ms * 1e-3) / 1e9 / pk["hbm_gbs"],
            "compaction_128_images_gbs": big_bytes / (big_ms * 1e-3) / 1e9,
            "compaction_128_images_hbm_frac": big_bytes / (big_ms * 1e-3) / 1e9 / pk["hbm_gbs"],
            "compaction_note": ("16-image figures: one call after an L2 flush, events around it (launch latency "
                                "included); 128 images: 402 MB moved per call, back to back"),
            "roofline_attention": attention_roofline(attn_full_ms, attn_full_flops, m.n_layers, pk, workloads),
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
                       "ms_per_step_pruned_prefix_cuda_graph": dec_graph_ms,
                       "hbm_frac_pruned_cuda_graph": ((weight_bytes + cache_bytes(pruned_lens)) / (dec_graph_ms * 1e-3)
                                                      / 1e9 / pk["hbm_gbs"]) if dec_graph_ms else None,
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
            "workloads": workloads,
            "scaling_table": scaling,
        }
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


# ----------------------------------------------------------------------------- per-workload measurements

def device_selector_weights(s, dev, gen, torch):
    """Selector weights drawn on the device (timing only), with the
    distributions of synth.make_selector_weights: N(0, 0.02) matrices (bf16 for
    the encoder and the text projection, fp32 for the pointer decoder), unit
    LayerNorm gains and zero biases."""
    def bf(shape):
        return (torch.randn(shape, device=dev, generator=gen) * 0.02).to(torch.bfloat16)

    def f32(shape):
        return torch.randn(shape, device=dev, generator=gen) * 0.02

    def ones(n):
        return torch.ones(n, device=dev)

    def zeros(n):
        return torch.zeros(n, device=dev)

    D, Dt, h, F = s.D, s.D_text, s.h, s.enc_ffn
    out = {"W_p": bf((D, Dt)), "ln_text_g": ones(D), "ln_text_b": zeros(D), "enc": [],
           "s_stop": f32((D,)), "s_start": f32((D,)), "W_in": f32((h, D)), "ln1_g": ones(h), "ln1_b": zeros(h),
           "ln2_g": ones(h), "ln2_b": zeros(h), "Wk_p": f32((h, D))}
    for n in ("Wq_s", "Wk_s", "Wv_s", "Wo_s", "Wq_p"):
        out[n] = f32((h, h))
    for _ in range(s.n_enc_layers):
        out["enc"].append({"ln1_g": ones(D), "ln1_b": zeros(D), "Wqkv": bf((3 * D, D)), "Wo": bf((D, D)),
                           "ln2_g": ones(D), "ln2_b": zeros(D), "W1": bf((F, D)), "W2": bf((D, F))})
    return out


def device_model(B, m, dev, gen, torch, max_pos):
    layers = [device_layer_weights(m, l, dev, gen, torch) for l in range(m.n_layers)]
    head = {"final_norm": torch.ones(m.d, device=dev), "proj_W1": None, "proj_W2": None}
    if m.proj_kind == "linear":
        head["proj_W1"] = (torch.randn((m.d, m.proj_in), device=dev, generator=gen) * 0.02).to(torch.bfloat16)
    elif m.proj_kind == "mlp2":
        head["proj_W1"] = (torch.randn((m.proj_hidden, m.proj_in), device=dev, generator=gen) * 0.02).to(torch.bfloat16)
        head["proj_W2"] = (torch.randn((m.d, m.proj_hidden), device=dev, generator=gen) * 0.02).to(torch.bfloat16)
    return B.Model(m, layers, head, dev, max_pos=max_pos)


def attention_roofline(ms, flops, layers, pk, workloads):
    """The attention kernels against the dense bf16 peak (burst: the launches
    are timed one by one): the full prefix of the 16-image batch (16 x 624
    tokens, the head-pair kernel) and, when the per-workload pass ran, the
    InternVL3 full prefix (4 x 3,424 tokens, GQA 28/4, the two-stream kernel)."""
    achieved = flops / (ms * 1e-3) / 1e12
    out = {"kernel": "attn_pair_kernel (tcgen05; sequences up to 1,280 tokens)", "bound": "tensor",
           "workload": "llava15-7b-b16 full prefix: 16 x 624 tokens, 32 heads of 128, causal",
           "achieved": achieved, "peak": pk["bf16"], "unit": "TFLOP/s", "frac": achieved / pk["bf16"],
           "peak_source": pk["source"] + " bf16 burst", "traffic": attn_traffic(),
           "traffic_unit": "DRAM bytes per launch (one layer)", "launches": layers,
           "algorithmic": "4 H d_h sum L(L+1)/2 flops per layer (causal)"}
    w = (workloads or {}).get("internvl3-tiles-b4")
    if isinstance(w, dict) and w.get("full_prefix"):
        fp = w["full_prefix"]
        out["long"] = {"kernel": "attn_fa_kernel (tcgen05, two softmax streams, dynamic scheduling)",
                       "workload": "internvl3-tiles-b4 full prefix: 4 x 3,424 tokens, GQA 28/4, 28 layers",
                       "achieved": fp.get("attention_tflops"), "frac": fp.get("attention_frac_of_bf16_burst")}
    return out


def attn_flops(m, lens, causal=True):
    """Algorithmic attention flops of one layer: 4 H d_h sum L(L+1)/2 causal,
    4 H d_h sum L^2 bidirectional."""
    if causal:
        return 4.0 * m.n_heads * m.head_dim * sum(L * (L + 1) / 2 for L in lens)
    return 4.0 * m.n_heads * m.head_dim * sum(L * L for L in lens)


class Timing:
    """CUDA-event timers on the current stream (warmed, synchronised on both sides)."""

    def __init__(self, torch, dev):
        self.torch = torch
        self.flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)  # twice the L2

    def timed(self, fn, reps=3, warm=1):
        torch = self.torch
        for _ in range(warm):
            fn()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(reps):
            fn()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b) / reps

    def cold(self, fn, reps=5):
        """One call after an L2 flush, a spin kernel ahead so the host has
        enqueued the events and the call before the GPU reaches them."""
        torch = self.torch
        fn()
        total = 0.0
        for _ in range(reps):
            self.flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda._sleep(1_000_000)
            a.record()
            fn()
            b.record()
            torch.cuda.synchronize()
            total += a.elapsed_time(b)
        return total / reps

    def profiled(self, B, fn):
        """Per-kernel-kind event time of one call (events around every launch)."""
        B.sp_profile_begin(20000)
        fn()
        self.torch.cuda.synchronize()
        return B.sp_profile_end()


def measure_config(B, torch, tm, w, model, dev, gen, pk, *, targets, mean_target, reps=2):
    """One workload end to end on device-drawn weights and inputs: STOP biases
    calibrated for the targets; the whole pipeline; selection alone (us per
    image); compaction (GB/s, HBM fraction, one call after an L2 flush); the
    pruned prefill (compaction + projector + prefill) against the full-prefix
    prefill on the same kernels; GEMM and attention flop rates from per-launch
    events against the measured bf16 peak."""
    s, m = w.selector, w.model
    sel = B.Selector(s, device_selector_weights(s, dev, gen, torch), dev)
    X = torch.randn((sum(w.n_vis), s.D), device=dev, generator=gen).to(torch.bfloat16)
    E = (torch.randn((sum(w.n_txt), s.D_text), device=dev, generator=gen) * 0.02).to(torch.bfloat16)
    eps = w.episodes()
    n_ep = len(eps)
    cal = B.sp_select(sel, w.n_vis, w.n_txt, X=X, E_text=E, stop_bias=B.dev_f32(np.full(n_ep, -1e30), dev),
                      group_size=w.group_size, g=w.g, k_max=w.k_max)
    torch.cuda.synchronize()
    gaps, rounds = cal["gap"].cpu().numpy(), cal["rounds"].cpu().numpy()
    biases, _ = S.stop_biases([gaps[e, :rounds[e]] for e in range(n_ep)], targets, g=w.g, k_max=w.k_max,
                              n_cand=[n for (_, _, n) in eps], mean_target=mean_target)
    bias = B.dev_f32(biases, dev)
    pipe = B.Pipeline(sel, model, w.n_vis, w.n_txt, group_size=w.group_size, g=w.g, k_max=w.k_max)
    pipe_ms = tm.timed(lambda: pipe(X, E, bias), reps=reps, warm=2)
    assert int(pipe.err.item()) == 0
    counts = pipe.count.cpu().numpy().astype(int)
    T = int(pipe.cu[-1].item())
    K_sum = int(counts.sum())
    lens = [int(k) + t for k, t in zip(counts, w.n_txt)]
    sws = {}

    def select():
        r = B.sp_select(sel, w.n_vis, w.n_txt, X=X, E_text=E, stop_bias=bias, group_size=w.group_size, g=w.g,
                        k_max=w.k_max, traces=False, ws=sws.get("ws"))
        sws["ws"], sws["r"] = r["_ws"], r
    select_ms = tm.timed(select, reps=reps)
    proj = m.proj_kind != "none"
    comp = {}

    def compact(idx, count, kc, key, index_mode=False):
        comp[key] = B.sp_compact(w.n_vis, w.n_txt, X=X, text=E, idx=idx, count=count, k_cap=kc,
                                 projector_mode=proj and not index_mode, index_mode=proj and index_mode,
                                 out=comp.get(key))
        return comp[key]

    r = sws["r"]
    # the gather as its own kernel (the copy the pipeline folds into the projector's operand loads)
    compact_ms = tm.cold(lambda: compact(r["idx"], r["count"], pipe.k_cap, "c"))
    vis_w = s.D
    comp_bytes = 2.0 * (K_sum * vis_w + sum(w.n_txt) * m.d) * 2 + 4.0 * (w.B + 1 + T)
    st = {}

    def prefill_stage(idx, count, kc, key):
        o = compact(idx, count, kc, key, index_mode=True)
        if proj:
            B.sp_project(model, X=X, vis_src=o["vis_src"], vis_row_map=o["vis_row_map"], vis_cu=o["vis_cu"],
                         packed=o["packed"], rows_cap=o["rows_cap"], B=w.B, ws=st.get(key + "pw"))
        lens_cap = max(min(n, kc) + t for n, t in zip(w.n_vis, w.n_txt))
        res = B.sp_prefill(model, x=o["packed"], cu_seqlens=o["cu_seqlens"], pos=o["pos"], B=w.B, T_cap=o["T_cap"],
                           max_seqlen_cap=lens_cap, ws=st.get(key + "ws"), hidden=st.get(key + "h"))
        st[key + "ws"], st[key + "h"] = res["_ws"], res["hidden"]

    pruned_ms = tm.timed(lambda: prefill_stage(r["idx"], r["count"], pipe.k_cap, "p"), reps=reps)
    nmax = max(w.n_vis)
    full_idx = torch.full((w.B, nmax), -1, dtype=torch.int32, device=dev)
    for b, n in enumerate(w.n_vis):
        full_idx[b, :n] = torch.arange(n, dtype=torch.int32, device=dev)
    full_cnt = torch.tensor(w.n_vis, dtype=torch.int32, device=dev)
    full_ms = tm.timed(lambda: prefill_stage(full_idx, full_cnt, nmax, "f"), reps=reps)
    full_lens = [n + t for n, t in zip(w.n_vis, w.n_txt)]
    pf = tm.profiled(B, lambda: prefill_stage(full_idx, full_cnt, nmax, "f"))
    pp = tm.profiled(B, lambda: prefill_stage(r["idx"], r["count"], pipe.k_cap, "p"))
    pl = tm.profiled(B, lambda: pipe(X, E, bias))
    qkv = (m.n_heads + 2 * m.n_kv_heads) * m.head_dim
    p_lin = m.d * qkv + m.n_heads * m.head_dim * m.d + 3 * m.d * m.ffn
    proj_f = {"mlp2": m.proj_in * m.proj_hidden + m.proj_hidden * m.d, "linear": m.proj_in * m.d}.get(m.proj_kind, 0)

    def rates(prof, T_, K_, lens_):
        g_fl = 2.0 * (m.n_layers * p_lin * T_ + proj_f * K_)
        a_fl = m.n_layers * attn_flops(m, lens_)
        g_ms, a_ms = prof["gemm"]["ms"], prof["attention"]["ms"]
        return {"gemm_ms": g_ms, "gemm_tflops": g_fl / (g_ms * 1e-3) / 1e12 if g_ms else None,
                "gemm_frac_of_bf16_burst": g_fl / (g_ms * 1e-3) / 1e12 / pk["bf16"] if g_ms else None,
                "attention_ms": a_ms, "attention_tflops": a_fl / (a_ms * 1e-3) / 1e12 if a_ms else None,
                "attention_frac_of_bf16_burst": a_fl / (a_ms * 1e-3) / 1e12 / pk["bf16"] if a_ms else None}

    out = {"workload": w.name, "images": w.B, "visual_tokens": list(w.n_vis), "text_tokens": list(w.n_txt),
           "group_size": w.group_size, "g": w.g, "k_max": w.k_max, "layers": m.n_layers, "d": m.d,
           "heads": [m.n_heads, m.n_kv_heads], "kept": counts.tolist(), "mean_kept": float(counts.mean()),
           "packed_tokens": T, "full_tokens": sum(full_lens),
           "pipeline_ms": pipe_ms, "select_ms": select_ms, "select_us_per_image": 1e3 * select_ms / w.B,
           "compaction_ms": compact_ms, "compaction_gbs": comp_bytes / (compact_ms * 1e-3) / 1e9,
           "compaction_hbm_frac": comp_bytes / (compact_ms * 1e-3) / 1e9 / pk["hbm_gbs"],
           "pruned_prefill_ms": pruned_ms, "full_prefix_prefill_ms": full_ms,
           "speedup_prefill": full_ms / pruned_ms, "speedup_with_selection": full_ms / (pruned_ms + select_ms),
           "token_ratio": sum(full_lens) / T, "full_prefix": rates(pf, sum(full_lens), sum(w.n_vis), full_lens),
           "pruned": rates(pp, T, K_sum, lens),
           "pipeline_stages_ms": {k: v["ms"] for k, v in pl.items() if v["launches"]}}
    if m.n_layers == 1:
        wbytes = 2.0 * (p_lin + proj_f)
        out["weight_bytes"] = wbytes
        out["pruned_prefill_weight_gbs"] = wbytes / (pruned_ms * 1e-3) / 1e9
        out["pruned_prefill_hbm_frac"] = wbytes / (pruned_ms * 1e-3) / 1e9 / pk["hbm_gbs"]
    sel.close()
    return out


def episode_targets(w):
    """Kept-count targets per selection episode: the workload's statements
    (mean 64 for one 576-token image; AnyRes: 16..128 per tile group, mean 64,
    so 80..640 per image; Qwen: 11% of every group; InternVL: the mean kept)."""
    eps = w.episodes()
    if w.name.startswith("llavanext"):
        z = S.normal(w.seed, "group_targets", (len(eps),))
        t = np.clip(np.round(64 * np.exp(0.6 * z) / np.exp(0.6 * z).mean()), 16, 128).astype(int)
        return t, 64.0
    if w.name.startswith("qwen"):
        return np.array([max(1, int(round(0.11 * n))) for (_, _, n) in eps]), None
    return np.full(len(eps), int(w.target_mean_k)), float(w.target_mean_k)


def measure_workloads(B, torch, dev, gen, pk, c2_model, reps=2):
    """Every workload other than the headline one, and the InternVL STOP sweep."""
    tm = Timing(torch, dev)
    out = {}
    w1 = S.llava15_1layer()
    m1 = device_model(B, w1.model, dev, gen, torch, max_pos=1024)
    t, mt = episode_targets(w1)
    out["llava15-576-1layer"] = measure_config(B, torch, tm, w1, m1, dev, gen, pk, targets=t, mean_target=mt,
                                               reps=reps)
    m1.close()
    w3 = S.llavanext_anyres_b8()
    t, mt = episode_targets(w3)
    out["llavanext-anyres-b8"] = measure_config(B, torch, tm, w3, c2_model, dev, gen, pk, targets=t,
                                                mean_target=mt, reps=reps)
    w4 = S.qwen25vl_varres_b8()
    mq = device_model(B, w4.model, dev, gen, torch, max_pos=4096 + 256)
    t, mt = episode_targets(w4)
    out["qwen25vl-varres-b8"] = measure_config(B, torch, tm, w4, mq, dev, gen, pk, targets=t, mean_target=mt,
                                               reps=reps)
    sweep = []
    for k in (32, 64, 128, 256, 512):
        w5 = S.internvl3_tiles_b4(mean_k=k)
        t, mt = episode_targets(w5)
        r = measure_config(B, torch, tm, w5, mq, dev, gen, pk, targets=t, mean_target=mt, reps=reps)
        if k == 64:
            out["internvl3-tiles-b4"] = r
        sweep.append({"target_mean_kept": k, "mean_kept": r["mean_kept"], "select_us_per_image":
                      r["select_us_per_image"], "compaction_gbs": r["compaction_gbs"],
                      "pruned_prefill_ms": r["pruned_prefill_ms"], "full_prefix_prefill_ms": r["full_prefix_prefill_ms"],
                      "speedup_prefill": r["speedup_prefill"], "speedup_with_selection": r["speedup_with_selection"],
                      "pipeline_ms": r["pipeline_ms"]})
    out["internvl3_stop_sweep"] = sweep
    mq.close()
    return out


# Sec. 4 scaling table (LLaVA-1.5-7B rows): input tokens, retained tokens,
# full prefill ms, pruned-path ms, selector ms, on the paper's GPU (context only)
PAPER_SCALING = {
    320: (32, 29.34, 30.00, 9.65), 640: (64, 53.24, 37.14, 16.15), 960: (96, 70.86, 37.75, 20.45),
    1280: (128, 116.89, 40.91, 24.25), 1600: (160, 142.93, 46.13, 28.85), 1920: (192, 189.83, 52.28, 34.41),
    2240: (224, 236.55, 57.73, 39.14)}


def scaling_rows(B, torch, dev, gen, selector, model, steps, warmup):
    """Scaling with the visual-prefix length at 10% retention: one image of N
    visual + 48 text tokens on the LLaVA-1.5-7B-shaped model, N = 320..2240.
    Per N: the full-prefix prefill (projector on N rows + 32 layers over N + 48),
    the pruned path (selector incl. its encoder, compaction, projector on the
    kept rows, 32 layers over K + 48) and the selector alone, each the mean of
    `steps` calls after `warmup`."""
    L = 48
    tm = Timing(torch, dev)
    rows = []
    for N in sorted(PAPER_SCALING):
        K = N // 10
        X = (torch.randn((N, selector.shape.D), device=dev, generator=gen)).to(torch.bfloat16)
        E = (torch.randn((L, model.shape.d), device=dev, generator=gen) * 0.02).to(torch.bfloat16)
        bias = torch.full((1,), -1e30, dtype=torch.float32, device=dev)  # STOP never wins: exactly K kept
        pipe = B.Pipeline(selector, model, [N], [L], group_size=0, g=1, k_max=K)
        pruned_ms = tm.timed(lambda: pipe(X, E, bias), reps=steps, warm=warmup)
        sel_ws = {}

        def select():
            r = B.sp_select(selector, [N], [L], X=X, E_text=E, stop_bias=bias, group_size=0, g=1, k_max=K,
                            traces=False, ws=sel_ws.get("ws"))
            sel_ws["ws"] = r["_ws"]
        selector_ms = tm.timed(select, reps=steps, warm=warmup)
        full_idx = torch.arange(N, dtype=torch.int32, device=dev).reshape(1, N)
        full_cnt = torch.full((1,), N, dtype=torch.int32, device=dev)
        st = {}

        def full_prefill():
            o = B.sp_compact([N], [L], X=X, text=E, idx=full_idx, count=full_cnt, k_cap=N, index_mode=True,
                             out=st.get("c"))
            st["c"] = o
            B.sp_project(model, X=X, vis_src=o["vis_src"], vis_row_map=o["vis_row_map"], vis_cu=o["vis_cu"],
                         packed=o["packed"], rows_cap=o["rows_cap"], B=1)
            r = B.sp_prefill(model, x=o["packed"], cu_seqlens=o["cu_seqlens"], pos=o["pos"], B=1, T_cap=o["T_cap"],
                             max_seqlen_cap=N + L, ws=st.get("ws"), hidden=st.get("h"))
            st["ws"], st["h"] = r["_ws"], r["hidden"]
        full_ms = tm.timed(full_prefill, reps=steps, warm=warmup)
        kept = int(pipe.count[0].item())
        pk, pf, pp, ps = PAPER_SCALING[N]
        rows.append({"input_tokens": N, "retained": kept, "full_prefill_ms": full_ms, "stepprune_prefill_ms": pruned_ms,
                     "selector_ms": selector_ms, "speedup": full_ms / pruned_ms,
                     "selector_share": selector_ms / pruned_ms,
                     "paper": {"retained": pk, "full_prefill_ms": pf, "stepprune_prefill_ms": pp, "selector_ms": ps,
                               "speedup": pf / pp, "selector_share": ps / pp}})
        del pipe
    return rows


def run_sweep(args):
    """The scaling table alone (one JSON line, no headline)."""
    import torch
    from paper_2609_13804_gb300 import binding as B

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    w = S.llava15_7b_b16()
    s, m = w.selector, w.model
    selector = B.Selector(s, S.make_selector_weights(w), dev)
    gen = torch.Generator(device=dev)
    gen.manual_seed(w.seed)
    model = device_model(B, m, dev, gen, torch, max_pos=4096)
    rows = scaling_rows(B, torch, dev, gen, selector, model, args.steps, args.warmup)
    line = {"sweep": "visual-prefix length at 10% retention", "config": {"workload": "llava15-7b dims, 1 image",
            "text_tokens": 48, "layers": m.n_layers}, "steps": args.steps, "warmup": args.warmup,
            "paper_gpu": "RTX PRO 6000 Blackwell (the paper's; context only)", "rows": rows}
    print(json.dumps(line), flush=True)


def run_profile_case(case: str):
    """Small, self-contained invocations of one stage of the path, sized for
    `ncu --set full` captures (a few GB on the device at most, a handful of
    launches).  Shapes are those of the 16-image LLaVA-1.5-7B-shaped batch
    unless the case names another workload:

      gemm            1 decoder layer, T = 1791 (4 GEMMs)
      attention       1 decoder layer, like gemm
      attention_full  1 layer over the full prefix (16 x 624)
      attention_gqa   1 Qwen2.5-VL-dims layer (GQA 28/4) over 4 sequences of 3,424
      select          selection from a given memory H
      select_deep     2-layer pointer decoder, 4 images, cap 64
      compact         compaction of the batch
      compact_full    every visual token kept (50 MB)
      decode          4 decoder layers, 16 sequences, 3 steps

    Each case runs its stage twice (the second launch set is the one to capture
    with `-s`)."""
    import torch

    from paper_2609_13804_gb300 import binding as B

    dev = torch.device("cuda", 0)
    w = S.internvl3_tiles_b4() if case == "attention_gqa" else S.llava15_7b_b16()
    counts = S.target_counts(w)
    if case in ("gemm", "attention", "attention_full", "attention_gqa", "decode"):
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
        model = B.Model(m, None, None, dev, max_pos=4096, device_weights={"layers": layers, "head": head})
        lens = [int(k) + 48 for k in counts]
        if case in ("attention_full", "attention_gqa"):
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
        kc = max(w.n_vis) if case in ("attention_full", "attention_gqa") else w.k_max
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


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu", action="store_true", help="skip the CPU oracle baseline")
    ap.add_argument("--launch-list", action="store_true",
                    help="set up, warm up and run one more step only (for an ncu launch list)")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the other workloads, the InternVL STOP sweep and the scaling table")
    ap.add_argument("--profile-case", default=None,
                    help="run one small stage invocation for an ncu capture (see run_profile_case)")
    ap.add_argument("--sweep", action="store_true",
                    help="scaling with the visual-prefix length at 10%% retention (one JSON line, no headline)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.profile_case:
        run_profile_case(args.profile_case)
    elif args.sweep:
        run_sweep(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
