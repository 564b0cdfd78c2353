"""Writes bf16_envelope_llava15_7b_{2,32}layers.json: how far two exact
emulations of the same bf16 model drift apart over Llama-7B-dims layers, on the
inputs of the 2-layer and of the 32-layer GPU prefill tests.

Both emulations round the same activations to bf16 where a bf16 model stores
them (the oracle's store='bf16').  The reference accumulates in fp64 and keeps
the attention probabilities exact; the second makes the two arithmetic choices
of a bf16 tensor-core implementation: fp32 accumulation of the four
projections (acc='fp32') and bf16 attention probabilities as the P V operand
(p_store='bf16').  A rounding decision that flips between them is as
legitimate in one as in the other, so their distance is the scale of
disagreement such an implementation has with the reference at that depth.  Also
written: the distance of the bf16-storage oracle from the pure fp64 oracle.
Inputs are those of the GPU tests (seeded synthetic).  Calls only the oracle and
the seeded generators.

    python tests/golden/bf16_envelope.py [2layers|32layers]   (default: both)
"""
import dataclasses
import json
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

from oracle import core as O  # noqa: E402
from paper_2609_13804_gb300 import synth as S  # noqa: E402

HERE = os.path.dirname(os.path.abspath(__file__))


def stats(a, b):
    d = np.abs(a - b)
    return {"max_abs": float(d.max()), "mean_rel": float(d.mean() / np.abs(b).mean())}


def run(seqs, layer_fn, n_layers, m, final_gain):
    """seqs: {name: rows}; returns the three final-normed variants per sequence."""
    h = {v: {k: x.astype(np.float64) for k, x in seqs.items()} for v in ("ref", "alt", "f64")}
    t0 = time.time()
    for l in range(n_layers):
        L = layer_fn(l)
        for k in seqs:
            n = len(seqs[k])
            h["ref"][k] = O.prefill_layer(h["ref"][k], L, m, [0, n], np.arange(n), store="bf16")
            h["alt"][k] = O.prefill_layer(h["alt"][k], L, m, [0, n], np.arange(n), store="bf16", acc="fp32",
                                          p_store="bf16")
            h["f64"][k] = O.prefill_layer(h["f64"][k], L, m, [0, n], np.arange(n))
        print(f"layer {l} done, {time.time() - t0:.0f} s", flush=True)
    return {v: np.concatenate([O.final_norm(h[v][k], m, final_gain) for k in seqs]) for v in h}


def write(name, meta, out):
    res = dict(meta)
    res["bf16_fp32acc_bf16p_vs_bf16_fp64acc"] = stats(out["alt"], out["ref"])
    res["bf16_storage_vs_fp64"] = stats(out["ref"], out["f64"])
    res["command"] = "python tests/golden/bf16_envelope.py"
    with open(os.path.join(HERE, f"bf16_envelope_llava15_7b_{name}.json"), "w") as f:
        json.dump(res, f, indent=1)
    print(name, json.dumps(res, indent=1))


def two_layers():
    """test_prefill_llama7b_dims_2layers: layers 0, 1 with norm gains, four
    ragged sequences; attention never crosses a sequence, so each runs alone."""
    w = S.llava15_7b_b16()
    m = w.model
    lens = [112, 240, 64, 17]
    cu = np.concatenate([[0], np.cumsum(lens)])
    x = S.bf16_round(S.normal(w.seed, "packed", (int(cu[-1]), m.d), 0.5))
    layers = [S.make_layer_weights(w, l, norm_affine=True) for l in range(2)]
    head = S.make_model_head(w, norm_affine=True)
    seqs = {b: x[cu[b]:cu[b + 1]] for b in range(len(lens))}
    out = run(seqs, lambda l: layers[l], 2, m, head["final_norm"])
    write("2layers", {"workload": w.name, "layers": 2, "sequences": lens}, out)


def thirty_two_layers():
    """test_prefill_llava15_b16_32layers_sampled: the shortest and the longest
    of the 16 packed sequences, 32 layers without norm gains."""
    w = S.llava15_7b_b16()
    m = dataclasses.replace(w.model, proj_kind="none", proj_in=w.model.d)
    lens = [int(k) + 48 for k in S.target_counts(w)]
    cu = np.concatenate([[0], np.cumsum(lens)])
    x = S.bf16_round(S.normal(w.seed, "packed32", (int(cu[-1]), m.d), 0.5))
    picks = [int(np.argmin(lens)), int(np.argmax(lens))]
    seqs = {b: x[cu[b]:cu[b + 1]] for b in picks}
    out = run(seqs, lambda l: S.make_layer_weights(w, l), m.n_layers, m, None)
    write("32layers", {"workload": w.name, "layers": m.n_layers, "sequences": {str(b): lens[b] for b in picks}}, out)


if __name__ == "__main__":
    which = sys.argv[1] if len(sys.argv) > 1 else "all"
    if which in ("2layers", "all"):
        two_layers()
    if which in ("32layers", "all"):
        thirty_two_layers()
