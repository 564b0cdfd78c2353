"""StepPrune inference path -- CPU oracle (TEST INFRASTRUCTURE ONLY).

A plain, slow, fp64 restatement of what the inference path of StepPrune
(arXiv 2609.13804) computes, written from the paper:

  * text projection and cross-modal input encoder      (Sec. 3.2, Eq. 3)
  * candidate memory with the learned STOP row          (Sec. 3.2, "Learned STOP Action")
  * pointer decoder, one hard step per round            (Sec. 3.2, Eq. 4)
  * grouped execution, TopG per non-STOP round          (Sec. 3.5, Eq. 11)
  * Algorithm 1: loop, restore to native order, gather  (Algorithm 1; Sec. 3.3, last paragraph)
  * frozen projector and LM prefill over the packed prefix (Sec. 3.3-3.4; LM dims of the
    evaluated backbones, Sec. 4.1), with 1-D RoPE or the 3-D mRoPE of the Qwen2.5-VL
    backbone (Sec. 1)
  * the training-time continuous pathway, forward only: trajectory aggregation,
    soft count, SoftTopK polarisation, variance-preserving noise gate (Sec. 3.3,
    Eqs. 5-9)

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg may import
this module.  It shares no code with the CUDA library and imports nothing from
the package; inputs arrive as numpy arrays from the seeded generators.

Readings of points the paper leaves open are stated at each function (see the
'Reading' notes); the list is repeated in the design notes of the repository.

Parity status of each function:
  layer_norm, rms_norm, gelu, silu      pinned (torch.nn.functional, closed forms)
  attention                             pinned (torch scaled_dot_product_attention, brute force)
  text_projection, encoder              pinned (torch.nn.TransformerEncoderLayer, fp64; the
                                        bf16-storage variant against a torch.nn.functional
                                        composition rounding the same tensors)
  pointer logits / select_episode       pinned (brute-force from-scratch decoder; torch
                                        nn.MultiheadAttention decoder; deeper decoders against
                                        torch nn.TransformerDecoderLayer; history-free top-K
                                        special case, Eq. 1; invariants of Alg. 1 and Eq. 11)
  restore / compact                     pinned (hand-worked golden fixture; invariants)
  rope                                  pinned (rotation closed form, relative-position property)
  mrope, mrope_positions                pinned (equal components -> rope; componentwise
                                        relative positions; norm kept; pruned positions
                                        = the full sequence's rows, by a grid walk)
  round_bf16                            pinned (torch's float32 -> bfloat16 conversion)
  trajectory_aggregate                  pinned (closed forms of Eqs. 5-7 for a constant
                                        STOP probability; Sum_i s_i = Kbar at beta = 1)
  trajectory_episode                    pinned (its hard rollout equals select_episode
                                        with g = 1; scratch = incremental; tau -> 0 gives
                                        Kbar = hard count, s = beta^t at the chosen step)
  soft_topk                             pinned (the two-anchor transport has the closed
                                        form sigmoid((s_i - theta) 2 / tau) with
                                        Sum alpha = k, found by bisection; n = 2, k = 1
                                        logistic; tau -> 0 hard top-k)
  vp_gate                               pinned (alpha = 1 / 0 ends; variance preserved)
  decode_step, cache_from_prefill       pinned (equals the prefill over the extended
                                        sequences at the new positions, with and
                                        without bf16 storage)
  projector                             pinned (torch nn.Sequential Linear-GELU-Linear)
  prefill_layer, prefill                pinned (a Llama decoder layer composed from
                                        torch.nn.functional in fp64: rms_norm, linear,
                                        complex-rotation RoPE, sdpa with repeated kv
                                        heads, silu -- GQA, ragged, both halves with
                                        residuals, with and without bf16 storage; zero
                                        output weights -> identity; uniform attention;
                                        varlen isolation and causality; acc='fp32'
                                        variant against acc='fp64' to fp32 precision)
  prefill_layer_rows                    pinned (equals prefill_layer at the chosen rows,
                                        1-D and 3-D positions, with and without storage
                                        rounding)
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence

import numpy as np
from scipy.special import erf as _erf

F64 = np.float64
NEG_INF = -np.inf


def _f(x) -> np.ndarray:
    return np.asarray(x, dtype=F64)


def round_bf16(x) -> np.ndarray:
    """Round to the nearest bfloat16 (ties to even), returned as fp64.

    bfloat16 keeps the top 16 bits of the IEEE fp32 pattern: the value is first
    rounded to fp32, then the low 16 bits are rounded away (ties to even)."""
    u = np.ascontiguousarray(_f(x).astype(np.float32)).view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    return r.astype(np.uint32).view(np.float32).astype(F64)


def _store(x, store: Optional[str]) -> np.ndarray:
    """Storage rounding of an activation between two ops: none (fp64 throughout)
    or 'bf16' (what a bf16 model keeps in memory between its kernels)."""
    if store is None:
        return _f(x)
    if store == "bf16":
        return round_bf16(x)
    raise ValueError(store)


# ----------------------------------------------------------------------------
# elementary layers
# ----------------------------------------------------------------------------

def layer_norm(x, eps: float, gain=None, bias=None) -> np.ndarray:
    """LayerNorm over the last axis, biased variance: (x - mu) / sqrt(var + eps) * g + b."""
    x = _f(x)
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    y = (x - mu) / np.sqrt(var + eps)
    if gain is not None:
        y = y * _f(gain)
    if bias is not None:
        y = y + _f(bias)
    return y


def rms_norm(x, eps: float, gain=None) -> np.ndarray:
    """RMSNorm over the last axis: x / sqrt(mean(x^2) + eps) * g."""
    x = _f(x)
    y = x / np.sqrt((x * x).mean(axis=-1, keepdims=True) + eps)
    if gain is not None:
        y = y * _f(gain)
    return y


def gelu(x) -> np.ndarray:
    """Exact GELU, x * Phi(x) = 0.5 x (1 + erf(x / sqrt 2))."""
    x = _f(x)
    return 0.5 * x * (1.0 + _erf(x / math.sqrt(2.0)))


def silu(x) -> np.ndarray:
    x = _f(x)
    return x / (1.0 + np.exp(-x))


def softmax(x, axis: int = -1) -> np.ndarray:
    x = _f(x)
    m = np.max(x, axis=axis, keepdims=True)
    e = np.exp(x - m)
    return e / e.sum(axis=axis, keepdims=True)


def attention(q, k, v, n_heads: int, n_kv_heads: int, causal: bool, q_pos=None,
              p_store: Optional[str] = None) -> np.ndarray:
    """Scaled dot-product attention of one sequence.

    q [Lq, Hq*dh], k/v [L, Hkv*dh].  Query head i reads key/value head
    floor(i * Hkv / Hq) (grouped-query attention; Hkv == Hq is plain MHA).
    Causal: the query at position p attends to key positions 0..p.  The query
    rows are the positions 0..L-1 of the sequence unless q_pos gives their
    positions (a subset of the sequence's rows).  p_store='bf16' rounds the
    attention probabilities to bf16 before they weight the values (the operand
    precision of a bf16 tensor-core P V product).
    """
    q, k, v = _f(q), _f(k), _f(v)
    Lq, L = q.shape[0], k.shape[0]
    dh = q.shape[1] // n_heads
    out = np.zeros((Lq, n_heads * dh), dtype=F64)
    mask = np.zeros((Lq, L), dtype=F64)
    if causal:
        qp = np.arange(Lq) if q_pos is None else np.asarray(q_pos, dtype=np.int64)
        mask[np.arange(L)[None, :] > qp[:, None]] = NEG_INF
    for i in range(n_heads):
        j = (i * n_kv_heads) // n_heads
        qi = q[:, i * dh:(i + 1) * dh]
        kj = k[:, j * dh:(j + 1) * dh]
        vj = v[:, j * dh:(j + 1) * dh]
        s = qi @ kj.T / math.sqrt(dh) + mask
        out[:, i * dh:(i + 1) * dh] = _store(softmax(s, axis=-1), p_store) @ vj
    return out


# ----------------------------------------------------------------------------
# selector: text projection and cross-modal encoder (Sec. 3.2, Eq. 3)
# ----------------------------------------------------------------------------

def text_projection(E_text, sel: Dict, eps: float, g_text: float = 1.0) -> np.ndarray:
    """E~_text = g_text * LN(W_p E_text) (Sec. 3.2).  Rows of E_text are tokens.

    Reading: g_text = 1 at inference (it is only ramped during training).
    """
    P = _f(E_text) @ _f(sel["W_p"]).T
    return g_text * layer_norm(P, eps, sel.get("ln_text_g"), sel.get("ln_text_b"))


def encoder_block(x, L: Dict, n_heads: int, eps: float, store: Optional[str] = None) -> np.ndarray:
    """One pre-norm ViT block with bidirectional self-attention (Sec. 3.2; the
    bidirectional mask is the default of Table 7(a)).

    Reading: no linear biases; MLP is W2 GELU(W1 x) with exact GELU.  The
    residual stream stays fp64; with store='bf16' the activations a bf16 model
    keeps between ops (normalised inputs, q / k / v, attention output, GELU
    output) are rounded to bf16 where they are stored.
    """
    x = _f(x)
    D = x.shape[1]
    a = _store(layer_norm(x, eps, L.get("ln1_g"), L.get("ln1_b")), store)
    qkv = _store(a @ _f(L["Wqkv"]).T, store)
    o = attention(qkv[:, :D], qkv[:, D:2 * D], qkv[:, 2 * D:], n_heads, n_heads, causal=False)
    x = x + _store(o, store) @ _f(L["Wo"]).T
    m = _store(layer_norm(x, eps, L.get("ln2_g"), L.get("ln2_b")), store)
    x = x + _store(gelu(m @ _f(L["W1"]).T), store) @ _f(L["W2"]).T
    return x


def encoder(X, E_tilde, sel: Dict, n_heads: int, eps: float, store: Optional[str] = None) -> np.ndarray:
    """H = Enc([X; E~_text])_[1:N] (Eq. 3): joint encoding, visual rows kept.

    Reading: the blocks are followed by no final norm.
    """
    X = _f(X)
    x = np.concatenate([X, _f(E_tilde)], axis=0)
    for L in sel["enc"]:
        x = encoder_block(x, L, n_heads, eps, store)
    return x[:X.shape[0]]


# ----------------------------------------------------------------------------
# pointer decoder (Sec. 3.2, Eq. 4) and grouped execution (Sec. 3.5, Eq. 11)
# ----------------------------------------------------------------------------
#
# Reading of the decoder the paper leaves unspecified (layer count, width):
#   one pre-LN decoder layer of width h with single-head attention.  A decoder
#   token is W_in q_t, where q_1 = s_start and q_{t+1} = M[a_t] is the hard
#   forward value of M^T p~_t.  Causal self-attention over the history gives
#     u_t = y_t + Wo_s * sum_i softmax_i(<Wq_s x_t, Wk_s x_i> / sqrt h) Wv_s x_i,
#     x_i = LN1(y_i),
#   and the pointer logits are the cross-attention scores of that layer:
#     l_t(j) = <Wq_p LN2(u_t), Wk_p M_j> / sqrt h,  j in 1..N+1 (N+1 = STOP).
#   In the last layer the cross-attention values and the FFN do not feed the
#   logits, so they are not computed.  The STOP logit gets an extra per-episode
#   stop_bias (the knob that sets the mean retained count of random-init models).
#
# Deeper decoders (dec["lower"], one dict per layer before the last): each such
#   layer is a whole pre-LN decoder layer of width h (Sec. 3.2: causal
#   self-attention over the history, cross-attention to the memory M, a
#   feed-forward network), its output the next layer's input:
#     a = x + Wo_s SelfAttn(LN1(x))          causal, single head, 1/sqrt h
#     c = a + Wo_c CrossAttn(LN2(a), M)      all N+1 rows of M (the mask acts on
#                                            the pointer logits only)
#     x' = c + W2 GELU(W1 LN3(c))            hidden width 4h, exact-erf GELU as in
#                                            the encoder blocks
#   and the top-level weights describe the last layer, as for one layer.

def decoder_tokens(rows, dec: Dict) -> np.ndarray:
    """Decoder input tokens y = W_in m for rows m in the D-wide memory space."""
    return _f(rows) @ _f(dec["W_in"]).T


def decoder_full_layer(X, M, L: Dict, eps: float) -> np.ndarray:
    """One full decoder layer (a layer before the last) over a whole history X
    [t, h]: causal self-attention, cross-attention to every row of M, FFN."""
    X = _f(X)
    h = X.shape[1]
    t = X.shape[0]
    x1 = layer_norm(X, eps, L.get("ln1_g"), L.get("ln1_b"))
    S = (x1 @ _f(L["Wq_s"]).T) @ (x1 @ _f(L["Wk_s"]).T).T / math.sqrt(h)
    S[np.triu_indices(t, 1)] = NEG_INF
    a = X + (softmax(S, axis=-1) @ (x1 @ _f(L["Wv_s"]).T)) @ _f(L["Wo_s"]).T
    x2 = layer_norm(a, eps, L.get("ln2_g"), L.get("ln2_b"))
    Sc = (x2 @ _f(L["Wq_c"]).T) @ (_f(M) @ _f(L["Wk_c"]).T).T / math.sqrt(h)
    c = a + (softmax(Sc, axis=-1) @ (_f(M) @ _f(L["Wv_c"]).T)) @ _f(L["Wo_c"]).T
    x3 = layer_norm(c, eps, L.get("ln3_g"), L.get("ln3_b"))
    return c + gelu(x3 @ _f(L["W1"]).T) @ _f(L["W2"]).T


def pointer_keys(M, dec: Dict) -> np.ndarray:
    """Cross-attention keys Wk_p M_j of all N+1 candidates."""
    return _f(M) @ _f(dec["Wk_p"]).T


def pointer_logits_from_scratch(history_rows, M, dec: Dict, eps: float) -> np.ndarray:
    """Raw pointer logits l_t over all N+1 rows of M, recomputing the whole
    decoder over the history [q_1, ..., q_t] (no cached state)."""
    h = dec["W_in"].shape[0]
    Y = decoder_tokens(history_rows, dec)
    for L in dec.get("lower", []):
        Y = decoder_full_layer(Y, M, L, eps)
    X1 = layer_norm(Y, eps, dec.get("ln1_g"), dec.get("ln1_b"))
    Q = X1 @ _f(dec["Wq_s"]).T
    K = X1 @ _f(dec["Wk_s"]).T
    V = X1 @ _f(dec["Wv_s"]).T
    t = Y.shape[0]
    S = Q @ K.T / math.sqrt(h)
    S[np.triu_indices(t, 1)] = NEG_INF
    U = Y + (softmax(S, axis=-1) @ V) @ _f(dec["Wo_s"]).T
    query = layer_norm(U[-1], eps, dec.get("ln2_g"), dec.get("ln2_b")) @ _f(dec["Wq_p"]).T
    return pointer_keys(M, dec) @ query / math.sqrt(h)


class _IncrementalDecoder:
    """The same decoder with the history's keys and values cached; each step
    adds the new tokens and evaluates only the last position."""

    def __init__(self, M, dec: Dict, eps: float):
        self.dec, self.eps = dec, eps
        self.h = dec["W_in"].shape[0]
        self.Kp = pointer_keys(M, dec)
        self.Y: List[np.ndarray] = []      # inputs of the last layer
        self.Ks: List[np.ndarray] = []
        self.Vs: List[np.ndarray] = []
        # layers before the last: their self-attention caches and the memory's
        # cross-attention keys / values
        self.lower = list(dec.get("lower", []))
        self.lK: List[List[np.ndarray]] = [[] for _ in self.lower]
        self.lV: List[List[np.ndarray]] = [[] for _ in self.lower]
        self.cK = [_f(M) @ _f(L["Wk_c"]).T for L in self.lower]
        self.cV = [_f(M) @ _f(L["Wv_c"]).T for L in self.lower]

    def _through_lower(self, y):
        """The new position through every layer before the last."""
        x, h, e = y, self.h, self.eps
        for i, L in enumerate(self.lower):
            x1 = layer_norm(x, e, L.get("ln1_g"), L.get("ln1_b"))
            self.lK[i].append(x1 @ _f(L["Wk_s"]).T)
            self.lV[i].append(x1 @ _f(L["Wv_s"]).T)
            att = softmax(np.stack(self.lK[i]) @ (x1 @ _f(L["Wq_s"]).T) / math.sqrt(h))
            a = x + (att @ np.stack(self.lV[i])) @ _f(L["Wo_s"]).T
            x2 = layer_norm(a, e, L.get("ln2_g"), L.get("ln2_b"))
            ca = softmax(self.cK[i] @ (x2 @ _f(L["Wq_c"]).T) / math.sqrt(h))
            c = a + (ca @ self.cV[i]) @ _f(L["Wo_c"]).T
            x3 = layer_norm(c, e, L.get("ln3_g"), L.get("ln3_b"))
            x = c + gelu(x3 @ _f(L["W1"]).T) @ _f(L["W2"]).T
        return x

    def append(self, rows):
        d = self.dec
        for y in decoder_tokens(np.atleast_2d(rows), d):
            y = self._through_lower(y)
            x = layer_norm(y, self.eps, d.get("ln1_g"), d.get("ln1_b"))
            self.Y.append(y)
            self.Ks.append(x @ _f(d["Wk_s"]).T)
            self.Vs.append(x @ _f(d["Wv_s"]).T)

    def logits(self) -> np.ndarray:
        d, h = self.dec, self.h
        y = self.Y[-1]
        x = layer_norm(y, self.eps, d.get("ln1_g"), d.get("ln1_b"))
        q = x @ _f(d["Wq_s"]).T
        a = softmax(np.stack(self.Ks) @ q / math.sqrt(h))
        u = y + (a @ np.stack(self.Vs)) @ _f(d["Wo_s"]).T
        query = layer_norm(u, self.eps, d.get("ln2_g"), d.get("ln2_b")) @ _f(d["Wq_p"]).T
        return self.Kp @ query / math.sqrt(h)


def select_episode(H, dec: Dict, *, k_max: int, g: int = 1, stop_bias: float = 0.0,
                   eps: float = 1e-5, mode: str = "incremental",
                   force: Optional[Sequence[int]] = None) -> Dict:
    """Algorithm 1, steps 2-3, over one candidate memory.

    H: [N, D] encoded visual candidates; M = [H; s_stop] (STOP is row N).
    Each round: l_r = PtrAttn(q_r, M) + Mask_r (+ stop_bias on STOP).
      * STOP wins when its logit is strictly above every still-available visual
        logit (ties go to the lower index, and STOP has the highest index);
        the round is counted and the episode ends.
      * Otherwise U_r = TopG of the available visual logits (Eq. 11), ordered by
        (logit desc, index asc), truncated to k_max - |S|; U_r joins S, is
        masked, and its rows M[U_r] join the causal history in that order.
      * The loop ends without another evaluation once |S| = k_max (reading of the
        cap: the paper's T_max counts steps, the workloads state a token cap).
      * With every visual candidate taken, only STOP is left and wins.

    Returns the step-order selection, its count, and per evaluated round:
    'margin' (smallest gap between consecutive values among the top g+1 of the
    available visual logits and STOP: the sensitivity of the round's decision)
    and 'gap' (best available visual logit minus the raw STOP logit, before
    stop_bias).

    force: teacher forcing along another implementation's step-order list.
    Each round takes the next min(g, k_max - |S|, #available) forced indices in
    the forced order instead of its own TopG, and STOP once the list is used up
    (with candidates left and |S| < k_max); the logits are those of the forced
    history.  'slack' then holds, per evaluated round, how far the forced
    decision is from one this oracle could take: the largest of (the take-th
    best available logit minus the lowest forced logit), (the STOP logit minus
    the best available logit: STOP is checked once per round, against the
    round's best), the largest rise between consecutive forced logits, and for
    a forced STOP (the best available logit minus the STOP logit); 0 when the
    forced decision is an exact optimum.
    """
    H = _f(H)
    N = H.shape[0]
    M = np.concatenate([H, _f(dec["s_stop"])[None, :]], axis=0)
    stop = N
    taken = np.zeros(N, dtype=bool)
    S: List[int] = []
    margins: List[float] = []
    gaps: List[float] = []
    stopped = False
    history = [_f(dec["s_start"])]
    inc = None
    if mode == "incremental":
        inc = _IncrementalDecoder(M, dec, eps)
        inc.append(history[0])
    elif mode != "scratch":
        raise ValueError(mode)

    slacks: List[float] = []
    while len(S) < k_max:
        if inc is not None:
            raw = inc.logits()
        else:
            raw = pointer_logits_from_scratch(np.stack(history), M, dec, eps)
        logits = raw.copy()
        logits[stop] += stop_bias
        logits[:N][taken] = NEG_INF
        avail = np.flatnonzero(~taken)
        if avail.size == 0:
            gaps.append(NEG_INF)
            margins.append(np.inf)
            slacks.append(0.0)
            stopped = True
            break
        vis = logits[avail]
        # candidates ranked by (logit desc, index asc); STOP ranks after equal visual logits
        rank = np.lexsort((avail, -vis))
        best = vis[rank[0]]
        gaps.append(float(best - raw[stop]))
        top = sorted([float(v) for v in vis[rank[:g + 1]]] + [float(logits[stop])], reverse=True)
        top = top[:g + 1]
        margins.append(min((top[i] - top[i + 1] for i in range(len(top) - 1)), default=np.inf))
        take = min(g, k_max - len(S), avail.size)
        if force is not None:
            if len(S) == len(force):
                slacks.append(max(0.0, float(best - logits[stop])))
                stopped = True
                break
            U = [int(a) for a in force[len(S):len(S) + take]]
            if len(U) < take or len(set(U)) < take or any(taken[u] for u in U):
                raise ValueError("forced actions: too few, repeated or already taken")
            lu = logits[U]
            slacks.append(max(0.0, float(vis[rank[take - 1]] - lu.min()), float(logits[stop] - best),
                              max((float(lu[i + 1] - lu[i]) for i in range(take - 1)), default=0.0)))
        else:
            if logits[stop] > best:
                stopped = True
                break
            U = [int(avail[i]) for i in rank[:take]]
        S.extend(U)
        taken[U] = True
        if inc is not None:
            inc.append(M[U])
        else:
            history.extend(M[U])
    out = {"order": S, "count": len(S), "margin": margins, "gap": gaps,
           "rounds": len(margins), "stopped": stopped}
    if force is not None:
        if len(S) != len(force):
            raise ValueError("forced list longer than the cap allows")
        out["slack"] = slacks
    return out


def restore(S: Sequence[int]) -> np.ndarray:
    """Algorithm 1 step 4: the retained indices in native visual order."""
    return np.sort(np.asarray(S, dtype=np.int64))


def select_image(H_b, dec: Dict, *, k_max: int, g: int, group_size: int,
                 stop_bias: Sequence[float], eps: float = 1e-5,
                 mode: str = "incremental") -> Dict:
    """Selection over one image whose candidates may be split into groups.

    Reading (candidate groups; the paper's 'grouped' means g tokens per round):
    each contiguous group of group_size candidates is an independent episode with
    its own mask, history and cap, the shared s_start / s_stop, and its own
    stop_bias entry; the image keeps the union of the groups' selections,
    offset to image positions and restored to native order.  group_size 0 means
    one episode over the whole image.
    """
    H_b = _f(H_b)
    N = H_b.shape[0]
    gs = group_size if group_size > 0 else N
    starts = list(range(0, N, gs))
    if len(stop_bias) != len(starts):
        raise ValueError("one stop_bias per episode")
    eps_out, idx = [], []
    for e, s in enumerate(starts):
        r = select_episode(H_b[s:s + gs], dec, k_max=k_max, g=g, stop_bias=float(stop_bias[e]),
                           eps=eps, mode=mode)
        eps_out.append(r)
        idx.extend(s + i for i in r["order"])
    return {"idx": restore(idx), "count": len(idx), "episodes": eps_out}


# ----------------------------------------------------------------------------
# training-time continuous pathway, forward only (Sec. 3.3: Eqs. 5-9)
# ----------------------------------------------------------------------------
#
# Reading (rollout): the hard rollout is Eq. 4 exactly as at inference with one
# token per step (the grouped rounds of Sec. 3.5 are an inference device): it
# ends at the first hard STOP, at K_max kept tokens, or with only STOP left.
# p_t = softmax(l_t / tau) is taken at every evaluated step (masked slots get
# probability 0, STOP is the last slot, stop_bias enters l_t(STOP) as at
# inference: pass 0 for the paper's training), and the sums of Eqs. 6-7 run over
# those steps; steps after the end of the rollout contribute nothing.


def trajectory_aggregate(P, beta: float) -> Dict:
    """Eqs. 5-7 over the evaluated steps of one rollout.

    P: [T, N+1] pointer distributions of steps t = 1..T (STOP in the last column).
      A_1 = 1,  A_t = prod_{u<t} (1 - p_u(STOP))                     (Eq. 5)
      s_i = sum_t A_t p_t(i) beta^t                                   (Eq. 6)
      Kbar = sum_t A_t (1 - p_t(STOP))                                (Eq. 7)
    """
    P = _f(P)
    T, n1 = P.shape
    s = np.zeros(n1 - 1, dtype=F64)
    kbar = 0.0
    A = 1.0
    alive = []
    for t in range(1, T + 1):
        p = P[t - 1]
        alive.append(A)
        s += A * p[:-1] * beta ** t
        kbar += A * (1.0 - p[-1])
        A *= 1.0 - p[-1]
    return {"s": s, "kbar": kbar, "alive": np.asarray(alive)}


def trajectory_episode(H, dec: Dict, *, k_max: int, tau: float, beta: float, stop_bias: float = 0.0,
                       eps: float = 1e-5, mode: str = "incremental",
                       force: Optional[Sequence[int]] = None, force_stop: Optional[bool] = None) -> Dict:
    """The training-time rollout of one episode (Eq. 4 with g = 1) and its
    aggregates (Eqs. 5-7).

    Each step: l_t = PtrAttn(q_t, M) + Mask_t (+ stop_bias on STOP),
    p_t = softmax(l_t / tau), a_t = argmax_j l_t(j) (lowest index on ties, so
    STOP, the last slot, wins only when strictly above every available visual
    logit); a visual a_t is masked and M[a_t] (the forward value of M^T p~_t)
    joins the causal history.

    force / force_stop: teacher forcing -- the actions taken are force[0..] and
    then STOP iff force_stop (a rollout of another implementation replayed to
    compare the distributions along it); the argmax is not consulted.
    """
    H = _f(H)
    N = H.shape[0]
    M = np.concatenate([H, _f(dec["s_stop"])[None, :]], axis=0)
    stop = N
    taken = np.zeros(N, dtype=bool)
    S: List[int] = []
    P: List[np.ndarray] = []
    stopped = False
    history = [_f(dec["s_start"])]
    inc = None
    if mode == "incremental":
        inc = _IncrementalDecoder(M, dec, eps)
        inc.append(history[0])
    elif mode != "scratch":
        raise ValueError(mode)
    while len(S) < k_max:
        if force is not None and len(S) == len(force) and not force_stop:
            break
        raw = inc.logits() if inc is not None else pointer_logits_from_scratch(np.stack(history), M, dec, eps)
        logits = raw.copy()
        logits[stop] += stop_bias
        logits[:N][taken] = NEG_INF
        P.append(softmax(logits / tau))
        avail = np.flatnonzero(~taken)
        if avail.size == 0:
            stopped = True
            break
        if force is not None:
            if len(S) == len(force):
                stopped = True
                break
            a = int(force[len(S)])
            if taken[a]:
                raise ValueError("forced action already taken")
        else:
            best = avail[np.argmax(logits[avail])]  # argmax returns the lowest index among equals
            if logits[stop] > logits[best]:
                stopped = True
                break
            a = int(best)
        S.append(a)
        taken[a] = True
        if inc is not None:
            inc.append(M[a])
        else:
            history.append(M[a])
    agg = trajectory_aggregate(np.stack(P), beta) if P else {"s": np.zeros(N), "kbar": 0.0, "alive": np.zeros(0)}
    return {"order": S, "count": len(S), "stopped": stopped, "rounds": len(P), "P": np.stack(P) if P else None,
            "s": agg["s"], "kbar": agg["kbar"], "alive": agg["alive"]}


def soft_topk(s, k: float, tau: float, tol: float = 1e-13, max_iter: int = 1_000_000) -> np.ndarray:
    """Eq. 8's SoftTopK_{k,tau}(s), which the paper only cites (the optimal-
    transport top-k of Xie et al., 2020).

    Reading: the entropic optimal transport of the n scores (mass 1/n each) onto
    two anchors y = (0, 1) with masses ((n - k)/n, k/n), cost (s_i - y_j)^2 and
    entropic regularisation tau; alpha_i = n Gamma_i,2, the share of token i sent
    to the "kept" anchor.  Solved here by Sinkhorn's alternating scaling in the
    log domain until the row marginals are met to `tol` (the column marginals
    are exact after each column update).  k <= 0 gives all zeros and k >= n all
    ones (the transport plan is then fixed by the marginals alone).
    """
    s = _f(s).ravel()
    n = s.size
    if n == 0:
        return np.zeros(0)
    if k <= 0:
        return np.zeros(n)
    if k >= n:
        return np.ones(n)
    y = np.array([0.0, 1.0])
    C = (s[:, None] - y[None, :]) ** 2
    log_mu = np.full(n, -math.log(n))
    log_nu = np.log(np.array([(n - k) / n, k / n]))

    def lse(x, axis):
        m = np.max(x, axis=axis, keepdims=True)
        return (m + np.log(np.sum(np.exp(x - m), axis=axis, keepdims=True))).squeeze(axis)

    f = np.zeros(n)
    g = np.zeros(2)
    for _ in range(max_iter):
        f = tau * (log_mu - lse((g[None, :] - C) / tau, axis=1))
        g = tau * (log_nu - lse((f[:, None] - C) / tau, axis=0))
        G = np.exp((f[:, None] + g[None, :] - C) / tau)
        if np.max(np.abs(G.sum(axis=1) * n - 1.0)) < tol:
            break
    else:
        raise RuntimeError("Sinkhorn did not converge")
    return n * G[:, 1]


def vp_gate(x, alpha, noise) -> np.ndarray:
    """Eq. 9: x~_i = sqrt(alpha_i) x_i + sqrt(1 - alpha_i) eps_i, one alpha per
    token (row); the Gaussian draws eps are an input."""
    a = _f(alpha)[:, None]
    return np.sqrt(a) * _f(x) + np.sqrt(1.0 - a) * _f(noise)


def train_forward(H, n_vis: Sequence[int], dec: Dict, *, k_max: int, group_size: int, tau: float,
                  beta: float, topk_tau: float, stop_bias: Sequence[float], X=None, noise=None,
                  eps: float = 1e-5, mode: str = "incremental", forced: Optional[Sequence] = None) -> Dict:
    """The continuous training pathway over a batch, forward only.

    Per episode (an image, or one candidate group of it): trajectory_episode.
    Per image: s = its episodes' scores at image positions, Kbar_b = the sum of
    its episodes' soft counts.  Eq. 8: k = the batch mean of Kbar_b (detached;
    the same k for every image, clamped to [0, N_b] per image), alpha_b =
    SoftTopK_{k, topk_tau}(s_b).  Eq. 9 when X and noise are given.
    forced: per episode (order, stopped) to replay instead of the argmax.
    """
    H = _f(H)
    offs = np.concatenate([[0], np.cumsum(n_vis)]).astype(int)
    s_all = np.zeros(offs[-1])
    kbar_ep, kbar_img, eps_out = [], [], []
    e = 0
    for b, n in enumerate(n_vis):
        gs = group_size if group_size > 0 else n
        kb = 0.0
        for c0 in range(0, n, gs):
            f = forced[e] if forced is not None else (None, None)
            r = trajectory_episode(H[offs[b] + c0: offs[b] + min(c0 + gs, n)], dec, k_max=k_max, tau=tau,
                                   beta=beta, stop_bias=float(stop_bias[e]), eps=eps, mode=mode,
                                   force=f[0], force_stop=f[1])
            s_all[offs[b] + c0: offs[b] + c0 + len(r["s"])] = r["s"]
            kbar_ep.append(r["kbar"])
            kb += r["kbar"]
            eps_out.append(r)
            e += 1
        kbar_img.append(kb)
    k = float(np.mean(kbar_img))
    alpha = np.zeros(offs[-1])
    for b, n in enumerate(n_vis):
        alpha[offs[b]:offs[b + 1]] = soft_topk(s_all[offs[b]:offs[b + 1]], min(max(k, 0.0), n), topk_tau)
    out = {"s": s_all, "kbar": np.asarray(kbar_ep), "kbar_image": np.asarray(kbar_img), "k": k,
           "alpha": alpha, "episodes": eps_out}
    if X is not None and noise is not None:
        out["x_gated"] = vp_gate(X, alpha, noise)
    return out


# ----------------------------------------------------------------------------
# compaction, projector, LM prefill
# ----------------------------------------------------------------------------

def compact(X, n_vis: Sequence[int], idx_list: Sequence[Sequence[int]], text, n_txt: Sequence[int]):
    """Algorithm 1 step 5 plus the LM input layout: per image the gathered visual
    rows X_b[idx_b] (native order) followed by the image's text rows.

    Reading: positions restart at 0 for every sequence (1-D RoPE of the LLaVA /
    Llama convention), and the visual prefix precedes the text (Sec. 3.3-3.4).
    Returns the packed rows, cu_seqlens [B+1] and positions [T].
    """
    X, text = _f(X), _f(text)
    rows, lens = [], []
    v0 = t0 = 0
    for b in range(len(n_vis)):
        Xb = X[v0:v0 + n_vis[b]]
        sel = np.asarray(idx_list[b], dtype=np.int64)
        rows.append(Xb[sel])
        rows.append(text[t0:t0 + n_txt[b]])
        lens.append(len(sel) + n_txt[b])
        v0 += n_vis[b]
        t0 += n_txt[b]
    packed = np.concatenate(rows, axis=0) if rows else np.zeros((0, X.shape[1]))
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    pos = np.concatenate([np.arange(n) for n in lens]).astype(np.int64) if lens else np.zeros(0, np.int64)
    return packed, cu, pos


def projector(rows, head: Dict, store: Optional[str] = None) -> np.ndarray:
    """Frozen multimodal projector applied to the kept visual rows after the
    restore (Sec. 3.3): linear W1 x, or the two-layer W2 GELU(W1 x).  With
    store='bf16' the hidden activation and the output are stored as bf16."""
    kind = head["proj_kind"]
    rows = _f(rows)
    if kind == "none":
        return rows
    if kind == "linear":
        return _store(rows @ _f(head["proj_W1"]).T, store)
    if kind == "mlp2":
        a = _store(gelu(rows @ _f(head["proj_W1"]).T), store)
        return _store(a @ _f(head["proj_W2"]).T, store)
    raise ValueError(kind)


def rope(x, pos, n_heads: int, head_dim: int, theta: float) -> np.ndarray:
    """Rotate-half rotary embedding: in every head, pair (i, i + dh/2) is rotated
    by angle pos * theta^(-2i/dh)."""
    x = _f(x).reshape(x.shape[0], n_heads, head_dim)
    half = head_dim // 2
    inv = theta ** (-(2.0 * np.arange(half, dtype=F64)) / head_dim)
    ang = _f(pos)[:, None] * inv[None, :]
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    a, b = x[..., :half], x[..., half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1).reshape(x.shape[0], -1)


def mrope(x, pos3, n_heads: int, head_dim: int, theta: float, section: Sequence[int]) -> np.ndarray:
    """Three-dimensional multimodal rotary embedding (the mRoPE of the
    Qwen2.5-VL backbone the method is evaluated on, Sec. 1 and Sec. 4.1).

    Reading: the dh/2 rotation pairs of every head are cut into consecutive
    sections of section[0], section[1], section[2] pairs (temporal, height,
    width); pair i of section c is rotated (rotate-half, as `rope`) by angle
    pos3[:, c] * theta^(-2i/dh), i counted over all dh/2 pairs.
    """
    x = _f(x).reshape(x.shape[0], n_heads, head_dim)
    half = head_dim // 2
    if sum(section) != half:
        raise ValueError("mRoPE sections must cover the dh/2 pairs")
    comp = np.repeat(np.arange(3), section)
    inv = theta ** (-(2.0 * np.arange(half, dtype=F64)) / head_dim)
    ang = _f(pos3)[:, comp] * inv[None, :]
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    a, b = x[..., :half], x[..., half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1).reshape(x.shape[0], -1)


def mrope_positions(kept, n_vis: int, grid_w: int, n_txt: int) -> np.ndarray:
    """(t, h, w) positions of one packed sequence [kept visual tokens; text].

    Reading (Sec. 3.3, last paragraph: the kept tokens are restored to native
    order so the backbone's positional convention holds): the image's N tokens
    form a grid of ceil(N / grid_w) rows of grid_w tokens at time 0; a kept
    token keeps its grid position (0, row, column); the text after the image
    continues, on all three components, from the largest position of the whole
    (unpruned) image block plus one, as it would without pruning.  So every
    row of the pruned sequence has the position it has in the full sequence.
    """
    kept = np.asarray(kept, dtype=np.int64)
    gh = -(-n_vis // grid_w)
    vis = np.stack([np.zeros_like(kept), kept // grid_w, kept % grid_w], axis=1)
    start = max(gh, grid_w)
    txt = np.repeat((start + np.arange(n_txt))[:, None], 3, axis=1)
    return np.concatenate([vis, txt], axis=0).astype(F64)


def _rotary(x, pos, n_heads: int, m) -> np.ndarray:
    """rope for 1-D positions, mrope (the model's sections) for [rows, 3] ones."""
    if np.ndim(pos) == 2:
        return mrope(x, pos, n_heads, m.head_dim, m.rope_theta, m.mrope_section)
    return rope(x, pos, n_heads, m.head_dim, m.rope_theta)


def _mm(a, b, acc: str) -> np.ndarray:
    """a @ b with fp64 arithmetic, or (acc='fp32') with fp32 operands and an
    fp32 result, the precision of a tensor-core product's accumulator."""
    if acc == "fp64":
        return a @ b
    if acc == "fp32":
        return (np.asarray(a, np.float32) @ np.asarray(b, np.float32)).astype(F64)
    raise ValueError(acc)


def prefill_layer(h, L: Dict, m, cu: Sequence[int], pos, store: Optional[str] = None,
                  acc: str = "fp64", kv_out: Optional[list] = None, p_store: Optional[str] = None) -> np.ndarray:
    """One pre-norm decoder layer of the frozen LM over the packed sequences:
    h += Wo Attn(RoPE(Wq x), RoPE(Wk x), Wv x), x = RMSNorm(h);
    h += Wdown (SiLU(Wg x') * Wu x'), x' = RMSNorm(h).  Attention is causal and
    never crosses a sequence boundary.  The residual stream h stays fp64; with
    store='bf16' the activations a bf16 model keeps between ops (normalised
    inputs, rotated q / k, v, attention output, SwiGLU output) are rounded to
    bf16 where they are stored.  acc='fp32' computes the four projections in
    fp32 instead of fp64 (used only to size how far two exact bf16 prefills
    drift apart through rounding decisions alone; p_store='bf16' likewise
    rounds the attention probabilities).  kv_out, if given, receives
    this layer's (rotated keys, values) of every packed row: the cache a
    generation step reads."""
    h = _f(h).copy()
    Hq, Hkv, dh, F = m.n_heads, m.n_kv_heads, m.head_dim, m.ffn
    x = _store(rms_norm(h, m.rms_eps, L.get("attn_norm")), store)
    qkv = _mm(x, _f(L["Wqkv"]).T, acc)
    q = _store(_rotary(qkv[:, :Hq * dh], pos, Hq, m), store)
    k = _store(_rotary(qkv[:, Hq * dh:(Hq + Hkv) * dh], pos, Hkv, m), store)
    v = _store(qkv[:, (Hq + Hkv) * dh:], store)
    if kv_out is not None:
        kv_out.append((k.copy(), v.copy()))
    o = np.zeros((h.shape[0], Hq * dh), dtype=F64)
    for b in range(len(cu) - 1):
        s, e = int(cu[b]), int(cu[b + 1])
        if e > s:
            o[s:e] = attention(q[s:e], k[s:e], v[s:e], Hq, Hkv, causal=True, p_store=p_store)
    h = h + _mm(_store(o, store), _f(L["Wo"]).T, acc)
    x2 = _store(rms_norm(h, m.rms_eps, L.get("mlp_norm")), store)
    gu = _mm(x2, _f(L["Wgu"]).T, acc)
    h = h + _mm(_store(silu(gu[:, :F]) * gu[:, F:], store), _f(L["Wdown"]).T, acc)
    return h


def prefill_layer_rows(h, L: Dict, m, cu: Sequence[int], pos, rows, store: Optional[str] = None) -> np.ndarray:
    """prefill_layer's output at the packed rows `rows` only (for sequences of
    thousands of tokens, where the whole layer is too slow for this oracle).

    Every step of the layer is row-local except the attention, whose query at
    position p reads the keys and values 0..p of its own sequence.  So the keys
    and values are projected (and rotated) for every row of the sequences the
    chosen rows lie in, while the queries, the attention, the output projection,
    the residuals and the MLP are evaluated for the chosen rows alone, in the
    same order, with the same storage rounding as prefill_layer.  Returns
    [len(rows), d] in the order of `rows`."""
    h = _f(h)
    rows = np.asarray(rows, dtype=np.int64)
    cu = np.asarray(cu, dtype=np.int64)
    Hq, Hkv, dh, F = m.n_heads, m.n_kv_heads, m.head_dim, m.ffn
    Wqkv = _f(L["Wqkv"])
    Wq, Wk, Wv = Wqkv[:Hq * dh], Wqkv[Hq * dh:(Hq + Hkv) * dh], Wqkv[(Hq + Hkv) * dh:]
    seq = np.searchsorted(cu, rows, side="right") - 1
    out = np.zeros((len(rows), h.shape[1]), dtype=F64)
    for b in np.unique(seq):
        s, e = int(cu[b]), int(cu[b + 1])
        sel = np.flatnonzero(seq == b)
        r = rows[sel]
        x = _store(rms_norm(h[s:e], m.rms_eps, L.get("attn_norm")), store)
        k = _store(_rotary(x @ Wk.T, pos[s:e], Hkv, m), store)
        v = _store(x @ Wv.T, store)
        q = _store(_rotary(x[r - s] @ Wq.T, pos[r], Hq, m), store)
        o = attention(q, k, v, Hq, Hkv, causal=True, q_pos=r - s)
        hr = h[r] + _store(o, store) @ _f(L["Wo"]).T
        x2 = _store(rms_norm(hr, m.rms_eps, L.get("mlp_norm")), store)
        gu = x2 @ _f(L["Wgu"]).T
        out[sel] = hr + _store(silu(gu[:, :F]) * gu[:, F:], store) @ _f(L["Wdown"]).T
    return out


def final_norm(h, m, gain=None) -> np.ndarray:
    """Output hidden states: RMSNorm of the last residual (the convention of
    returning the normalised last hidden state)."""
    return rms_norm(h, m.rms_eps, gain)


def prefill(x, layers: Sequence[Dict], m, cu, pos, final_gain=None, store: Optional[str] = None,
            acc: str = "fp64", kv_out: Optional[list] = None, p_store: Optional[str] = None) -> np.ndarray:
    h = _f(x)
    for L in layers:
        h = prefill_layer(h, L, m, cu, pos, store, acc, kv_out, p_store)
    return final_norm(h, m, final_gain)


def cache_from_prefill(kv_rows, cu) -> List[List[tuple]]:
    """Per layer, per sequence (K, V): the prefill's packed cache rows split at
    the sequence boundaries."""
    out = []
    for k, v in kv_rows:
        out.append([(k[int(cu[b]):int(cu[b + 1])].copy(), v[int(cu[b]):int(cu[b + 1])].copy())
                    for b in range(len(cu) - 1)])
    return out


def decode_step(x_new, layers: Sequence[Dict], m, cache: List[List[tuple]], final_gain=None,
                store: Optional[str] = None, rope_pos=None):
    """One generation step after the prefill over the pruned prefix (the decode
    the paper's per-token and end-to-end latencies include): sequence b's new
    token x_new[b] takes position len_b = cache rows of b and attends to the
    cached rotated keys / values 0..len_b-1 and to itself.  The layer is the
    prefill's layer applied to that one row.  Returns the normalised hidden
    state of the new tokens [B, d] and the cache with their keys / values
    appended.  rope_pos: the new tokens' rotary positions when they are not
    len_b (after an mRoPE prefix: generated text tokens have equal components,
    so their mRoPE is the 1-D rotation at that position)."""
    h = _f(x_new).copy()
    B = h.shape[0]
    Hq, Hkv, dh, F = m.n_heads, m.n_kv_heads, m.head_dim, m.ffn
    lens = [cache[0][b][0].shape[0] for b in range(B)]
    pos = np.array(lens if rope_pos is None else rope_pos, dtype=F64)
    new_cache = []
    for L, layer_cache in zip(layers, cache):
        x = _store(rms_norm(h, m.rms_eps, L.get("attn_norm")), store)
        qkv = x @ _f(L["Wqkv"]).T
        q = _store(rope(qkv[:, :Hq * dh], pos, Hq, dh, m.rope_theta), store)
        k = _store(rope(qkv[:, Hq * dh:(Hq + Hkv) * dh], pos, Hkv, dh, m.rope_theta), store)
        v = _store(qkv[:, (Hq + Hkv) * dh:], store)
        o = np.zeros((B, Hq * dh), dtype=F64)
        grown = []
        for b in range(B):
            Kb = np.concatenate([layer_cache[b][0], k[b:b + 1]])
            Vb = np.concatenate([layer_cache[b][1], v[b:b + 1]])
            grown.append((Kb, Vb))
            o[b] = attention(q[b:b + 1], Kb, Vb, Hq, Hkv, causal=False)[0]
        new_cache.append(grown)
        h = h + _store(o, store) @ _f(L["Wo"]).T
        x2 = _store(rms_norm(h, m.rms_eps, L.get("mlp_norm")), store)
        gu = x2 @ _f(L["Wgu"]).T
        h = h + _store(silu(gu[:, :F]) * gu[:, F:], store) @ _f(L["Wdown"]).T
    return final_norm(h, m, final_gain), new_cache


# ----------------------------------------------------------------------------
# the whole path (Algorithm 1 followed by the pruned prefill)
# ----------------------------------------------------------------------------

def run_pipeline(X, E_text, n_vis, n_txt, sel: Dict, sel_shape, head: Dict, layers, model_shape,
                 *, k_max: int, g: int, group_size: int, stop_bias: Sequence[float],
                 mode: str = "incremental", store: Optional[str] = None) -> Dict:
    """Selector encoder -> selection -> restore -> gather -> projector -> prefill."""
    X, E_text = _f(X), _f(E_text)
    n_heads = sel_shape.D // sel_shape.enc_head_dim
    idx_list, eps_per_img = [], []
    v0 = t0 = e0 = 0
    H_all = []
    for b in range(len(n_vis)):
        Et = text_projection(E_text[t0:t0 + n_txt[b]], sel, sel_shape.ln_eps, sel_shape.g_text)
        Hb = encoder(X[v0:v0 + n_vis[b]], Et, sel, n_heads, sel_shape.ln_eps)
        H_all.append(Hb)
        gs = group_size if group_size > 0 else n_vis[b]
        ne = (n_vis[b] + gs - 1) // gs
        r = select_image(Hb, sel, k_max=k_max, g=g, group_size=group_size,
                         stop_bias=stop_bias[e0:e0 + ne], eps=sel_shape.ln_eps, mode=mode)
        idx_list.append(r["idx"])
        eps_per_img.append(r)
        v0 += n_vis[b]
        t0 += n_txt[b]
        e0 += ne
    # gather (native order) then project the kept rows, then lay out [visual; text]
    v0 = 0
    vis_proj = []
    for b in range(len(n_vis)):
        vis_proj.append(projector(X[v0:v0 + n_vis[b]][idx_list[b]], head, store))
        v0 += n_vis[b]
    packed_rows, lens = [], []
    t0 = 0
    for b in range(len(n_vis)):
        packed_rows += [vis_proj[b], E_text[t0:t0 + n_txt[b]]]
        lens.append(len(idx_list[b]) + n_txt[b])
        t0 += n_txt[b]
    x = np.concatenate(packed_rows, axis=0)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    pos = np.concatenate([np.arange(n) for n in lens])
    hidden = prefill(x, layers, model_shape, cu, pos, head.get("final_norm"), store)
    return {"H": H_all, "idx": idx_list, "images": eps_per_img, "x": x, "cu_seqlens": cu,
            "pos": pos, "hidden": hidden}
