"""Seeded synthetic inputs and weights shared by the CUDA path's tests, the
oracle's tests and the benchmark.

This module holds no arithmetic of the method: it only draws numbers
(seeded PCG64 normals), rounds them to the storage types the path uses
(bf16 / fp32) and describes the workload shapes.  Everything it returns is
plain numpy, so the oracle and the CUDA binding can both consume it without
either importing the other.

Workload shapes follow the paper's four backbones (Sec. 4.1: LLaVA-1.5-7B with
576 visual tokens, LLaVA-NeXT-7B AnyRes with 2880, Qwen2.5-VL-7B dynamic
resolution, InternVL3-8B multi-tile) with random-init weights, because no
trained selector or MLLM weights are available.  The recipe (N(0, 1) visual
features, N(0, 0.02) text embeddings and weights) is the one stated next to each
shape below.
"""
from __future__ import annotations

import dataclasses
import hashlib
from typing import Dict, List, Optional

import numpy as np


# ----------------------------------------------------------------------------
# random numbers and storage rounding
# ----------------------------------------------------------------------------

def _subseed(seed: int, name: str) -> int:
    h = hashlib.sha256(f"{seed}/{name}".encode()).digest()
    return int.from_bytes(h[:8], "little")


def normal(seed: int, name: str, shape, std: float = 1.0) -> np.ndarray:
    """Seeded N(0, std^2) float32 array; the stream depends on (seed, name)."""
    g = np.random.Generator(np.random.PCG64(_subseed(seed, name)))
    return (g.standard_normal(size=shape, dtype=np.float32) * np.float32(std))


def uniform_int(seed: int, name: str, lo: int, hi: int, size) -> np.ndarray:
    g = np.random.Generator(np.random.PCG64(_subseed(seed, name)))
    return g.integers(lo, hi, size=size)


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round to nearest even."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    r = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32)


def bf16_round(x: np.ndarray) -> np.ndarray:
    """float32 values rounded to the nearest bf16 (returned as float32)."""
    return bf16_to_f32(bf16_bits(x))


# ----------------------------------------------------------------------------
# shapes
# ----------------------------------------------------------------------------

@dataclasses.dataclass
class SelectorShape:
    D: int            # visual feature width (candidate memory width)
    D_text: int       # text-embedding width (the LM width)
    h: int            # pointer-decoder width
    n_enc_layers: int = 2
    enc_head_dim: int = 64
    enc_ffn_mult: int = 4
    ln_eps: float = 1e-5
    g_text: float = 1.0
    n_dec_layers: int = 1  # pointer-decoder layers (the last one gives the logits)

    @property
    def enc_heads(self) -> int:
        return self.D // self.enc_head_dim

    @property
    def enc_ffn(self) -> int:
        return self.enc_ffn_mult * self.D


@dataclasses.dataclass
class ModelShape:
    n_layers: int
    d: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    rope_theta: float
    rms_eps: float
    proj_kind: str          # "none" | "linear" | "mlp2"
    proj_in: int            # visual width entering the projector
    proj_hidden: int        # hidden width of the 2-layer projector
    mrope_section: tuple = (0, 0, 0)  # rotation pairs per (t, h, w) component; zeros: 1-D RoPE


@dataclasses.dataclass
class Workload:
    name: str
    seed: int
    n_vis: List[int]        # visual tokens per image
    n_txt: List[int]        # text tokens per image
    selector: SelectorShape
    model: ModelShape
    group_size: int         # candidates per selection episode (0: whole image)
    g: int                  # tokens retained per non-STOP round
    k_max: int              # per-episode cap
    target_mean_k: float    # mean retained count the STOP bias is tuned for

    @property
    def B(self) -> int:
        return len(self.n_vis)

    def episodes(self):
        """(image, first candidate, candidate count) of every selection episode."""
        out = []
        for b, n in enumerate(self.n_vis):
            gs = self.group_size if self.group_size > 0 else n
            for s in range(0, n, gs):
                out.append((b, s, min(gs, n - s)))
        return out


def llava15_1layer(seed: int = 1001) -> Workload:
    """Single 576-token image, 32 text tokens, one 1024-wide decoder layer."""
    return Workload(
        name="llava15-576-1layer", seed=seed, n_vis=[576], n_txt=[32],
        selector=SelectorShape(D=1024, D_text=1024, h=256),
        model=ModelShape(n_layers=1, d=1024, n_heads=16, n_kv_heads=16, head_dim=64,
                         ffn=2816, rope_theta=1e4, rms_eps=1e-5, proj_kind="linear",
                         proj_in=1024, proj_hidden=1024),
        group_size=0, g=1, k_max=192, target_mean_k=64)


def llava15_7b_b16(seed: int = 1002) -> Workload:
    """16 x 576 visual tokens + 48 text tokens, Llama-7B dims, 32 layers."""
    return Workload(
        name="llava15-7b-b16", seed=seed, n_vis=[576] * 16, n_txt=[48] * 16,
        selector=SelectorShape(D=1024, D_text=4096, h=512),
        model=ModelShape(n_layers=32, d=4096, n_heads=32, n_kv_heads=32, head_dim=128,
                         ffn=11008, rope_theta=1e4, rms_eps=1e-5, proj_kind="mlp2",
                         proj_in=1024, proj_hidden=4096),
        group_size=0, g=1, k_max=192, target_mean_k=64)


def llavanext_anyres_b8(seed: int = 1003) -> Workload:
    """8 x 2880 visual tokens in 5 groups of 576, g=5, per-group cap 128."""
    return Workload(
        name="llavanext-anyres-b8", seed=seed, n_vis=[2880] * 8, n_txt=[64] * 8,
        selector=SelectorShape(D=1024, D_text=4096, h=512),
        model=ModelShape(n_layers=32, d=4096, n_heads=32, n_kv_heads=32, head_dim=128,
                         ffn=11008, rope_theta=1e4, rms_eps=1e-5, proj_kind="mlp2",
                         proj_in=1024, proj_hidden=4096),
        group_size=576, g=5, k_max=128, target_mean_k=320)


def qwen25vl_varres_b8(seed: int = 1004) -> Workload:
    """8 images with token counts drawn from {256,576,1024,2304,4096}, GQA 28/4."""
    sizes = np.array([256, 576, 1024, 2304, 4096])
    n_vis = [int(v) for v in sizes[uniform_int(seed, "n_vis", 0, 5, 8)]]
    return Workload(
        name="qwen25vl-varres-b8", seed=seed, n_vis=n_vis, n_txt=[64] * 8,
        selector=SelectorShape(D=3584, D_text=3584, h=512),
        model=ModelShape(n_layers=28, d=3584, n_heads=28, n_kv_heads=4, head_dim=128,
                         ffn=18944, rope_theta=1e6, rms_eps=1e-6, proj_kind="none",
                         proj_in=3584, proj_hidden=3584),
        group_size=1024, g=5, k_max=256, target_mean_k=0.11)


def internvl3_tiles_b4(seed: int = 1005, mean_k: int = 64) -> Workload:
    """4 images x (1 thumbnail + 12 tiles) x 256 = 3328 visual tokens, GQA 28/4."""
    return Workload(
        name=f"internvl3-tiles-b4-k{mean_k}", seed=seed, n_vis=[3328] * 4, n_txt=[96] * 4,
        selector=SelectorShape(D=3584, D_text=3584, h=512),
        model=ModelShape(n_layers=28, d=3584, n_heads=28, n_kv_heads=4, head_dim=128,
                         ffn=18944, rope_theta=1e6, rms_eps=1e-6, proj_kind="none",
                         proj_in=3584, proj_hidden=3584),
        group_size=0, g=5, k_max=1024, target_mean_k=mean_k)


WORKLOADS = {
    "llava15-576-1layer": llava15_1layer,
    "llava15-7b-b16": llava15_7b_b16,
    "llavanext-anyres-b8": llavanext_anyres_b8,
    "qwen25vl-varres-b8": qwen25vl_varres_b8,
    "internvl3-tiles-b4": internvl3_tiles_b4,
}


def tiny_workload(seed: int, n_vis, n_txt, D=32, D_text=48, h=16, d=64, n_heads=4,
                  n_kv_heads=2, head_dim=16, ffn=96, n_layers=2, group_size=0, g=1,
                  k_max=8, proj_kind="mlp2", enc_head_dim=16) -> Workload:
    """Small shapes for oracle self-tests and quick parity cases."""
    return Workload(
        name="tiny", seed=seed, n_vis=list(n_vis), n_txt=list(n_txt),
        selector=SelectorShape(D=D, D_text=D_text, h=h, enc_head_dim=enc_head_dim),
        model=ModelShape(n_layers=n_layers, d=d, n_heads=n_heads, n_kv_heads=n_kv_heads,
                         head_dim=head_dim, ffn=ffn, rope_theta=1e4, rms_eps=1e-5,
                         proj_kind=proj_kind, proj_in=D, proj_hidden=d),
        group_size=group_size, g=g, k_max=k_max, target_mean_k=k_max / 2)


# ----------------------------------------------------------------------------
# inputs and weights
# ----------------------------------------------------------------------------

def make_inputs(w: Workload) -> Dict[str, np.ndarray]:
    """Visual tokens X ~ N(0,1) (bf16) and text embeddings ~ N(0, 0.02) (bf16).

    E_text is given at the LM width D_text: it is both the prompt embedding the
    selector's text projection reads and the text rows of the LM input.
    """
    s = w.selector
    nv, nt = sum(w.n_vis), sum(w.n_txt)
    X = bf16_round(normal(w.seed, "X", (nv, s.D)))
    E = bf16_round(normal(w.seed, "E_text", (nt, s.D_text), 0.02))
    return {"X": X, "E_text": E}


def make_selector_weights(w: Workload, ln_affine: bool = False) -> Dict[str, object]:
    """Selector weights: bf16 encoder / text projection, fp32 pointer decoder.

    All matrices are N(0, 0.02) in nn.Linear layout [out, in]; s_start and s_stop
    are N(0, 0.02).  LayerNorm gains/biases are 1/0 unless ln_affine draws them.
    """
    s, seed = w.selector, w.seed
    D, Dt, h, F = s.D, s.D_text, s.h, s.enc_ffn

    def bf(name, shape):
        return bf16_round(normal(seed, name, shape, 0.02))

    def f32(name, shape, std=0.02):
        return normal(seed, name, shape, std)

    def ln(name, n):
        if not ln_affine:
            return np.ones(n, np.float32), np.zeros(n, np.float32)
        return (1.0 + normal(seed, name + ".g", (n,), 0.1)).astype(np.float32), \
            normal(seed, name + ".b", (n,), 0.1)

    out: Dict[str, object] = {}
    out["W_p"] = bf("sel.W_p", (D, Dt))
    out["ln_text_g"], out["ln_text_b"] = ln("sel.ln_text", D)
    enc = []
    for i in range(s.n_enc_layers):
        L = {}
        L["ln1_g"], L["ln1_b"] = ln(f"sel.enc{i}.ln1", D)
        L["Wqkv"] = bf(f"sel.enc{i}.Wqkv", (3 * D, D))
        L["Wo"] = bf(f"sel.enc{i}.Wo", (D, D))
        L["ln2_g"], L["ln2_b"] = ln(f"sel.enc{i}.ln2", D)
        L["W1"] = bf(f"sel.enc{i}.W1", (F, D))
        L["W2"] = bf(f"sel.enc{i}.W2", (D, F))
        enc.append(L)
    out["enc"] = enc
    out["s_stop"] = f32("sel.s_stop", (D,))
    out["s_start"] = f32("sel.s_start", (D,))
    out["W_in"] = f32("sel.W_in", (h, D))
    out["ln1_g"], out["ln1_b"] = ln("sel.dec.ln1", h)
    for n in ("Wq_s", "Wk_s", "Wv_s", "Wo_s", "Wq_p"):
        out[n] = f32("sel.dec." + n, (h, h))
    out["ln2_g"], out["ln2_b"] = ln("sel.dec.ln2", h)
    out["Wk_p"] = f32("sel.dec.Wk_p", (h, D))
    # decoder layers before the last (pointer decoders of n_dec_layers > 1);
    # the FFN matrices are bf16-representable (the GPU stores them as bf16)
    lower = []
    for i in range(getattr(s, "n_dec_layers", 1) - 1):
        L = {}
        L["ln1_g"], L["ln1_b"] = ln(f"sel.dec{i}.ln1", h)
        for n in ("Wq_s", "Wk_s", "Wv_s", "Wo_s", "Wq_c", "Wo_c"):
            L[n] = f32(f"sel.dec{i}.{n}", (h, h))
        L["Wk_c"] = f32(f"sel.dec{i}.Wk_c", (h, D))
        L["Wv_c"] = f32(f"sel.dec{i}.Wv_c", (h, D))
        L["ln2_g"], L["ln2_b"] = ln(f"sel.dec{i}.ln2", h)
        L["ln3_g"], L["ln3_b"] = ln(f"sel.dec{i}.ln3", h)
        L["W1"] = bf(f"sel.dec{i}.W1", (4 * h, h))
        L["W2"] = bf(f"sel.dec{i}.W2", (h, 4 * h))
        lower.append(L)
    if lower:
        out["lower"] = lower
    return out


def make_memory(w: Workload, name: str = "H") -> np.ndarray:
    """Candidate memory H [sum N_b, D] fp32 ~ N(0,1): input of the selection stage
    when it is exercised without the encoder."""
    return normal(w.seed, name, (sum(w.n_vis), w.selector.D))


def make_layer_weights(w: Workload, layer: int, norm_affine: bool = False) -> Dict[str, np.ndarray]:
    """One decoder layer of the LM: bf16 N(0, 0.02) weights in nn.Linear layout.

    Wqkv stacks [Wq; Wk; Wv] ([(Hq + 2 Hkv) dh, d]); Wgu stacks [W_gate; W_up]
    ([2F, d]).  RMSNorm gains are 1 unless norm_affine draws them.
    """
    m, seed = w.model, w.seed
    qkv = (m.n_heads + 2 * m.n_kv_heads) * m.head_dim

    def bf(name, shape):
        return bf16_round(normal(seed, f"lm{layer}.{name}", shape, 0.02))

    def gain(name):
        if not norm_affine:
            return np.ones(m.d, np.float32)
        return (1.0 + normal(seed, f"lm{layer}.{name}", (m.d,), 0.1)).astype(np.float32)

    return {
        "attn_norm": gain("attn_norm"),
        "Wqkv": bf("Wqkv", (qkv, m.d)),
        "Wo": bf("Wo", (m.d, m.n_heads * m.head_dim)),
        "mlp_norm": gain("mlp_norm"),
        "Wgu": bf("Wgu", (2 * m.ffn, m.d)),
        "Wdown": bf("Wdown", (m.d, m.ffn)),
    }


def make_model_head(w: Workload, norm_affine: bool = False) -> Dict[str, object]:
    """Projector and final norm of the LM."""
    m, seed = w.model, w.seed
    out: Dict[str, object] = {"proj_kind": m.proj_kind}
    if m.proj_kind == "linear":
        out["proj_W1"] = bf16_round(normal(seed, "proj.W1", (m.d, m.proj_in), 0.02))
    elif m.proj_kind == "mlp2":
        out["proj_W1"] = bf16_round(normal(seed, "proj.W1", (m.proj_hidden, m.proj_in), 0.02))
        out["proj_W2"] = bf16_round(normal(seed, "proj.W2", (m.d, m.proj_hidden), 0.02))
    out["final_norm"] = (np.ones(m.d, np.float32) if not norm_affine else
                         (1.0 + normal(seed, "final_norm", (m.d,), 0.1)).astype(np.float32))
    return out


def make_packed_lm_input(w: Workload, counts: List[int], name: str = "packed") -> Dict[str, np.ndarray]:
    """A packed prefill input (bf16 rows ~ N(0, 0.5)) with the sequence lengths
    counts[b] + n_txt[b]: the input of the prefill stage exercised on its own."""
    lens = [int(k) + int(t) for k, t in zip(counts, w.n_txt)]
    T = sum(lens)
    x = bf16_round(normal(w.seed, name, (T, w.model.d), 0.5))
    return {"x": x, "lens": np.array(lens, np.int64)}


def target_counts(w: Workload, n_episodes: Optional[int] = None) -> np.ndarray:
    """Per-image retained-count targets with the workload's mean.

    For a whole-image episode batch (llava15-7b-b16): spread 16..192 with mean
    64, lognormal in shape; the extremes are always present.
    """
    B = w.B
    if B == 1:
        return np.array([int(w.target_mean_k)])
    z = normal(w.seed, "k_targets", (B,))
    lo, hi, mean = 16, min(192, w.k_max), w.target_mean_k
    k = np.exp(0.7 * z)
    k = np.clip(np.round(k * mean / k.mean()), lo, hi).astype(np.int64)
    k[int(np.argmin(z))] = lo
    k[int(np.argmax(z))] = hi
    # nudge to the exact mean, one token at a time on the interior samples
    want = int(round(mean * B))
    i = 0
    order = np.argsort(z)
    inner = [j for j in order if k[j] not in (lo, hi)] or list(range(B))
    while k.sum() != want and i < 100000:
        j = inner[i % len(inner)]
        if k.sum() < want and k[j] < hi:
            k[j] += 1
        elif k.sum() > want and k[j] > lo:
            k[j] -= 1
        i += 1
    return k


# ----------------------------------------------------------------------------
# STOP-bias calibration of random-init selectors
# ----------------------------------------------------------------------------

def _realisable(gaps: np.ndarray):
    """Round counts a scalar STOP bias can produce for one episode, from its gap
    trace (best available visual logit minus raw STOP logit, recorded with STOP
    disabled): stopping after K rounds needs a bias above gap[K] and at or below
    every earlier gap, i.e. gap[K] must be a new running minimum."""
    R = len(gaps)
    out = [(0, float(gaps[0]) + 1.0 if R else 0.0)]
    run_min = np.inf
    for t in range(R):
        if t > 0 and gaps[t] < run_min:
            lo = float(gaps[t])
            bias = run_min - 1.0 if not np.isfinite(lo) else 0.5 * (lo + run_min)
            out.append((t, float(bias)))
        run_min = min(run_min, float(gaps[t]))
    if R:
        out.append((R, float(run_min) - 1.0 if np.isfinite(run_min) else -1e30))
    return out


def stop_biases(gap_traces, targets, *, g: int, k_max: int, n_cand, mean_target: Optional[float] = None):
    """Per-episode STOP biases whose kept counts are the realisable counts nearest
    to `targets` (tokens), then nudged so their mean approaches `mean_target`.

    gap_traces[e]: that episode's gap trace with STOP disabled; n_cand[e]: its
    candidate count.  Returns (biases float32, expected kept counts)."""
    opts = []
    for e, gaps in enumerate(gap_traces):
        gaps = np.asarray(gaps, np.float64)
        gaps = gaps[~np.isnan(gaps)]
        cand = []
        for rounds, bias in _realisable(gaps):
            cand.append((min(rounds * g, k_max, int(n_cand[e])), bias))
        opts.append(cand)
    pick = []
    for e, cand in enumerate(opts):
        pick.append(int(np.argmin([abs(k - targets[e]) for k, _ in cand])))
    if mean_target is not None:
        want = mean_target * len(opts)
        for _ in range(20 * len(opts)):
            tot = sum(opts[e][pick[e]][0] for e in range(len(opts)))
            best = None
            for e, cand in enumerate(opts):
                for step in (-1, 1):
                    j = pick[e] + step
                    if 0 <= j < len(cand):
                        nt = tot - cand[pick[e]][0] + cand[j][0]
                        gain = abs(tot - want) - abs(nt - want)
                        if gain > 0 and (best is None or gain > best[0]):
                            best = (gain, e, j)
            if best is None:
                break
            pick[best[1]] = best[2]
    biases = np.array([opts[e][pick[e]][1] for e in range(len(opts))], np.float32)
    counts = np.array([opts[e][pick[e]][0] for e in range(len(opts))], np.int64)
    return biases, counts
