"""Thin ctypes binding of libstepprune (include/stepprune.h).

Argument marshalling only: every computation runs in the library's CUDA
kernels.  PyTorch supplies device memory and streams.  The library is loaded on
first use; if it has not been built (paper_2609_13804_gb300.build) the call
raises instead of falling back to anything else.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Dict, List, Optional, Sequence

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libstepprune.so")

SP_MAX_BATCH = 256
SP_MAX_ENC_LAYERS = 4
SP_MAX_LM_LAYERS = 96
SP_MAX_KMAX = 1024
SP_MAX_NVIS = 16384

STATUS = {0: "SP_OK", 1: "SP_ERR_INVALID_ARG", 2: "SP_ERR_SHAPE", 3: "SP_ERR_ALIGN", 4: "SP_ERR_WORKSPACE",
          5: "SP_ERR_CUDA", 6: "SP_ERR_TIMEOUT", 7: "SP_ERR_UNSUPPORTED", 8: "SP_ERR_DEVICE"}
KERNEL_KINDS = ["gemm", "sgemm", "attention", "norm", "select", "restore", "compact", "misc", "train"]
PROJ = {"none": 0, "linear": 1, "mlp2": 2}

EXPORTS = [
    "sp_last_error", "sp_abi_version", "sp_device_error_status", "sp_selector_create", "sp_selector_destroy",
    "sp_num_episodes", "sp_select_workspace", "sp_select", "sp_packed_cap", "sp_compact", "sp_model_create",
    "sp_model_destroy", "sp_project_workspace", "sp_project", "sp_prefill_workspace", "sp_prefill",
    "sp_pipeline_workspace", "sp_pipeline", "sp_pipeline_host_workspace", "sp_pipeline_host",
    "sp_profile_begin", "sp_profile_end", "sp_select_noalloc",
    "sp_decode_workspace", "sp_decode", "sp_select_train", "sp_soft_topk", "sp_vp_gate",
    "sp_mrope_positions", "sp_wait_probe",
]
SP_SELECT_NOALLOC_SCRATCH_BYTES = 64 << 20

P = C.c_void_p
FP = C.POINTER(C.c_float)
IP = C.POINTER(C.c_int)


class sp_selector_cfg(C.Structure):
    _fields_ = [("D", C.c_int), ("D_text", C.c_int), ("h", C.c_int), ("n_enc_layers", C.c_int),
                ("enc_head_dim", C.c_int), ("enc_ffn", C.c_int), ("ln_eps", C.c_float), ("g_text", C.c_float),
                ("n_dec_layers", C.c_int)]


class sp_dec_layer_weights(C.Structure):
    _fields_ = [("ln1_g", P), ("ln1_b", P), ("Wq_s", P), ("Wk_s", P), ("Wv_s", P), ("Wo_s", P), ("ln2_g", P),
                ("ln2_b", P), ("Wq_c", P), ("Wo_c", P), ("Wk_c", P), ("Wv_c", P), ("ln3_g", P), ("ln3_b", P),
                ("W1", P), ("W2", P)]


class sp_selector_weights(C.Structure):
    _fields_ = [("W_p", P), ("ln_text_g", P), ("ln_text_b", P),
                ("enc_wqkv", P * SP_MAX_ENC_LAYERS), ("enc_wo", P * SP_MAX_ENC_LAYERS),
                ("enc_w1", P * SP_MAX_ENC_LAYERS), ("enc_w2", P * SP_MAX_ENC_LAYERS),
                ("enc_ln1_g", P * SP_MAX_ENC_LAYERS), ("enc_ln1_b", P * SP_MAX_ENC_LAYERS),
                ("enc_ln2_g", P * SP_MAX_ENC_LAYERS), ("enc_ln2_b", P * SP_MAX_ENC_LAYERS),
                ("s_stop", P), ("s_start", P), ("W_in", P), ("ln1_g", P), ("ln1_b", P),
                ("Wq_s", P), ("Wk_s", P), ("Wv_s", P), ("Wo_s", P), ("ln2_g", P), ("ln2_b", P),
                ("Wq_p", P), ("Wk_p", P), ("dec_lower", C.POINTER(sp_dec_layer_weights))]


class sp_select_in(C.Structure):
    _fields_ = [("B", C.c_int), ("n_vis", IP), ("n_txt", IP), ("X", P), ("E_text", P), ("H", P),
                ("stop_bias", P), ("group_size", C.c_int), ("g", C.c_int), ("k_max", C.c_int)]


class sp_select_out(C.Structure):
    _fields_ = [("idx", P), ("k_cap", C.c_int), ("count", P), ("order", P), ("ep_count", P),
                ("margin", P), ("gap", P), ("rounds", P), ("memory", P), ("err", P)]


class sp_train_args(C.Structure):
    _fields_ = [("tau", C.c_float), ("beta", C.c_float), ("score", P), ("kbar", P)]


class sp_compact_in(C.Structure):
    _fields_ = [("B", C.c_int), ("n_vis", IP), ("n_txt", IP), ("X", P), ("W_vis", C.c_int), ("text", P),
                ("W_txt", C.c_int), ("idx", P), ("k_cap", C.c_int), ("count", P)]


class sp_compact_out(C.Structure):
    _fields_ = [("packed", P), ("cu_seqlens", P), ("pos", P), ("vis_packed", P), ("vis_row_map", P),
                ("vis_cu", P), ("err", P), ("vis_src", P)]


class sp_model_cfg(C.Structure):
    _fields_ = [("n_layers", C.c_int), ("d", C.c_int), ("n_heads", C.c_int), ("n_kv_heads", C.c_int),
                ("head_dim", C.c_int), ("ffn", C.c_int), ("max_pos", C.c_int), ("rope_theta", C.c_float),
                ("rms_eps", C.c_float), ("proj_kind", C.c_int), ("proj_in", C.c_int), ("proj_hidden", C.c_int),
                ("mrope_section", C.c_int * 3)]


class sp_model_weights(C.Structure):
    _fields_ = [("wqkv", P * SP_MAX_LM_LAYERS), ("wo", P * SP_MAX_LM_LAYERS), ("wgu", P * SP_MAX_LM_LAYERS),
                ("wdown", P * SP_MAX_LM_LAYERS), ("attn_norm", P * SP_MAX_LM_LAYERS),
                ("mlp_norm", P * SP_MAX_LM_LAYERS), ("final_norm", P), ("proj_w1", P), ("proj_w2", P)]


class sp_project_io(C.Structure):
    _fields_ = [("B", C.c_int), ("rows_cap", C.c_int), ("vis_packed", P), ("vis_row_map", P), ("vis_cu", P),
                ("packed", P), ("err", P), ("X", P), ("rows_X", C.c_int), ("vis_src", P)]


class sp_prefill_io(C.Structure):
    _fields_ = [("B", C.c_int), ("T_cap", C.c_int), ("max_seqlen_cap", C.c_int), ("x", P), ("cu_seqlens", P),
                ("pos", P), ("hidden", P), ("residual", P), ("err", P), ("kv", P), ("kv_S_cap", C.c_int),
                ("pos3", P)]


class sp_decode_io(C.Structure):
    _fields_ = [("B", C.c_int), ("x", P), ("lens", P), ("kv", P), ("kv_S_cap", C.c_int), ("max_len_cap", C.c_int),
                ("hidden", P), ("err", P), ("rope_pos", P)]


class sp_pipeline_io(C.Structure):
    _fields_ = [("sel", sp_select_in), ("k_cap", C.c_int), ("idx", P), ("count", P), ("cu_seqlens", P),
                ("hidden", P), ("err", P)]


class sp_pipeline_host_io(C.Structure):
    _fields_ = [("sel", sp_select_in), ("k_cap", C.c_int), ("host_idx", P), ("host_count", P),
                ("host_cu_seqlens", P), ("host_hidden", P)]


_lib = None


def lib():
    """The loaded library (raises if it was not built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with `python -m paper_2609_13804_gb300.build`")
    L = C.CDLL(LIB_PATH)
    sig = {
        "sp_last_error": (C.c_char_p, []),
        "sp_abi_version": (C.c_int, []),
        "sp_device_error_status": (C.c_int, [C.c_int]),
        "sp_selector_create": (C.c_int, [C.POINTER(sp_selector_cfg), C.POINTER(sp_selector_weights), C.POINTER(P)]),
        "sp_selector_destroy": (None, [P]),
        "sp_num_episodes": (C.c_int, [C.c_int, IP, C.c_int]),
        "sp_select_workspace": (C.c_size_t, [P, C.POINTER(sp_select_in)]),
        "sp_select": (C.c_int, [P, C.POINTER(sp_select_in), C.POINTER(sp_select_out), P, C.c_size_t, P]),
        "sp_packed_cap": (C.c_int, [C.c_int, IP, IP, C.c_int]),
        "sp_compact": (C.c_int, [C.POINTER(sp_compact_in), C.POINTER(sp_compact_out), P]),
        "sp_model_create": (C.c_int, [C.POINTER(sp_model_cfg), C.POINTER(sp_model_weights), C.POINTER(P)]),
        "sp_model_destroy": (None, [P]),
        "sp_project_workspace": (C.c_size_t, [P, C.c_int]),
        "sp_project": (C.c_int, [P, C.POINTER(sp_project_io), P, C.c_size_t, P]),
        "sp_prefill_workspace": (C.c_size_t, [P, C.c_int, C.c_int]),
        "sp_prefill": (C.c_int, [P, C.POINTER(sp_prefill_io), P, C.c_size_t, P]),
        "sp_decode_workspace": (C.c_size_t, [P, C.c_int]),
        "sp_decode": (C.c_int, [P, C.POINTER(sp_decode_io), P, C.c_size_t, P]),
        "sp_pipeline_workspace": (C.c_size_t, [P, P, C.POINTER(sp_pipeline_io)]),
        "sp_pipeline": (C.c_int, [P, P, C.POINTER(sp_pipeline_io), P, C.c_size_t, P]),
        "sp_pipeline_host_workspace": (C.c_size_t, [P, P, C.POINTER(sp_pipeline_host_io)]),
        "sp_pipeline_host": (C.c_int, [P, P, C.POINTER(sp_pipeline_host_io), P, C.c_size_t, P]),
        "sp_select_noalloc": (C.c_int, [P, C.POINTER(sp_select_in), C.POINTER(sp_select_out), P]),
        "sp_select_train": (C.c_int, [P, C.POINTER(sp_select_in), C.POINTER(sp_select_out),
                                      C.POINTER(sp_train_args), P, C.c_size_t, P]),
        "sp_soft_topk": (C.c_int, [C.c_int, IP, C.c_int, P, P, C.c_float, P, P, P]),
        "sp_vp_gate": (C.c_int, [C.c_int, C.c_int, P, P, P, P, P]),
        "sp_mrope_positions": (C.c_int, [C.c_int, IP, IP, IP, P, C.c_int, P, P, C.c_int, P, P]),
        "sp_wait_probe": (C.c_int, [P, C.c_uint, C.c_int, P, P, P]),
        "sp_profile_begin": (C.c_int, [C.c_int]),
        "sp_profile_end": (C.c_int, [C.POINTER(C.c_double), C.POINTER(C.c_longlong), C.POINTER(C.c_double),
                                     C.POINTER(C.c_double)]),
    }
    for name, (res, args) in sig.items():
        f = getattr(L, name)
        f.restype = res
        f.argtypes = args
    _lib = L
    return L


class SPError(RuntimeError):
    pass


def _check(status: int, what: str):
    if status != 0:
        msg = lib().sp_last_error().decode(errors="replace")
        raise SPError(f"{what}: {STATUS.get(status, status)}: {msg}")


# ----------------------------------------------------------------------------- tensors

def _torch():
    import torch
    return torch


def ptr(t) -> Optional[int]:
    return None if t is None else t.data_ptr()


def dev_f32(a, device):
    torch = _torch()
    if isinstance(a, torch.Tensor):
        return a.to(device=device, dtype=torch.float32).contiguous()
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(device)


def dev_bf16(a, device):
    """bf16 device tensor holding exactly the values of `a` (which must already be
    bf16-representable, e.g. from synth.bf16_round)."""
    torch = _torch()
    if isinstance(a, torch.Tensor):
        return a.to(device=device, dtype=torch.bfloat16).contiguous()
    f = np.ascontiguousarray(a, dtype=np.float32)
    bits = (f.view(np.uint32) >> np.uint32(16)).astype(np.uint16)
    return torch.from_numpy(bits.view(np.int16)).to(device).view(torch.bfloat16)


def _int_array(v: Sequence[int]):
    arr = (C.c_int * len(v))(*[int(x) for x in v])
    return arr


def _stream(stream) -> Optional[int]:
    torch = _torch()
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def workspace(nbytes: int, device):
    torch = _torch()
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


# ----------------------------------------------------------------------------- selector

class Selector:
    """A selector handle plus the device copies of its weights (kept alive here)."""

    def __init__(self, shape, weights: Dict, device="cuda"):
        torch = _torch()
        self.shape, self.device = shape, torch.device(device)
        self._keep: List = []
        w = sp_selector_weights()

        def keep(t):
            self._keep.append(t)
            return ptr(t)

        nl = shape.n_enc_layers
        if nl > 0:
            w.W_p = keep(dev_bf16(weights["W_p"], device))
            w.ln_text_g = keep(dev_f32(weights["ln_text_g"], device))
            w.ln_text_b = keep(dev_f32(weights["ln_text_b"], device))
            for i, L in enumerate(weights["enc"]):
                w.enc_wqkv[i] = keep(dev_bf16(L["Wqkv"], device))
                w.enc_wo[i] = keep(dev_bf16(L["Wo"], device))
                w.enc_w1[i] = keep(dev_bf16(L["W1"], device))
                w.enc_w2[i] = keep(dev_bf16(L["W2"], device))
                w.enc_ln1_g[i] = keep(dev_f32(L["ln1_g"], device))
                w.enc_ln1_b[i] = keep(dev_f32(L["ln1_b"], device))
                w.enc_ln2_g[i] = keep(dev_f32(L["ln2_g"], device))
                w.enc_ln2_b[i] = keep(dev_f32(L["ln2_b"], device))
        for n in ("s_stop", "s_start", "W_in", "ln1_g", "ln1_b", "Wq_s", "Wk_s", "Wv_s", "Wo_s", "ln2_g",
                  "ln2_b", "Wq_p", "Wk_p"):
            setattr(w, n, keep(dev_f32(weights[n], device)))
        lower = weights.get("lower", [])
        nd = getattr(shape, "n_dec_layers", 1)
        if len(lower) != nd - 1:
            raise ValueError(f"{nd} decoder layers need {nd - 1} lower layers, got {len(lower)}")
        if lower:
            arr = (sp_dec_layer_weights * len(lower))()
            for i, L in enumerate(lower):
                for n in ("ln1_g", "ln1_b", "Wq_s", "Wk_s", "Wv_s", "Wo_s", "ln2_g", "ln2_b", "Wq_c", "Wo_c",
                          "Wk_c", "Wv_c", "ln3_g", "ln3_b"):
                    setattr(arr[i], n, keep(dev_f32(L[n], device)))
                arr[i].W1 = keep(dev_bf16(L["W1"], device))
                arr[i].W2 = keep(dev_bf16(L["W2"], device))
            self._keep.append(arr)
            w.dec_lower = C.cast(arr, C.POINTER(sp_dec_layer_weights))
        cfg = sp_selector_cfg(shape.D, shape.D_text, shape.h, nl, shape.enc_head_dim, shape.enc_ffn,
                              shape.ln_eps, shape.g_text, int(nd))
        h = P()
        _check(lib().sp_selector_create(C.byref(cfg), C.byref(w), C.byref(h)), "sp_selector_create")
        self.handle = h
        self._w = w

    def close(self):
        if getattr(self, "handle", None):
            lib().sp_selector_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def sp_num_episodes(n_vis, group_size: int) -> int:
    return lib().sp_num_episodes(len(n_vis), _int_array(n_vis), int(group_size))


def sp_packed_cap(n_vis, n_txt, k_cap: int) -> int:
    return lib().sp_packed_cap(len(n_vis), _int_array(n_vis), _int_array(n_txt), int(k_cap))


def k_cap_for(n_vis, group_size: int, k_max: int) -> int:
    """Largest possible kept count of one image (the minimum legal k_cap)."""
    best = 0
    for n in n_vis:
        gs = group_size if group_size > 0 else n
        best = max(best, sum(min(k_max, min(gs, n - s)) for s in range(0, n, gs)))
    return best


def _select_in(n_vis, n_txt, X, E_text, H, stop_bias, group_size, g, k_max, keep):
    nv, nt = _int_array(n_vis), _int_array(n_txt)
    keep += [nv, nt]
    return sp_select_in(len(n_vis), C.cast(nv, IP), C.cast(nt, IP), ptr(X), ptr(E_text), ptr(H), ptr(stop_bias),
                        int(group_size), int(g), int(k_max))


def sp_select(sel: Selector, n_vis, n_txt, *, stop_bias, X=None, E_text=None, H=None, group_size=0, g=1,
              k_max=192, k_cap=None, traces=True, memory=False, stream=None, ws=None,
              no_alloc=False, train=None) -> Dict:
    """Runs sp_select; returns device tensors idx [B, k_cap], count [B] and, with
    traces, order / ep_count / margin / gap / rounds / err.  no_alloc=True calls
    sp_select_noalloc instead (no workspace; the library's static scratch).
    train=(tau, beta) calls sp_select_train and adds score [sum N_b] and
    kbar [n_episodes] (the trajectory aggregates, Eqs. 5-7)."""
    torch = _torch()
    dev = sel.device
    keep: List = []
    inp = _select_in(n_vis, n_txt, X, E_text, H, stop_bias, group_size, g, k_max, keep)
    B = len(n_vis)
    E = sp_num_episodes(n_vis, group_size)
    if k_cap is None:
        k_cap = k_cap_for(n_vis, group_size, k_max)
    out = {"idx": torch.empty((B, k_cap), dtype=torch.int32, device=dev),
           "count": torch.empty(B, dtype=torch.int32, device=dev),
           "err": torch.zeros(1, dtype=torch.int32, device=dev)}
    if traces:
        out["order"] = torch.full((E, k_max), -1, dtype=torch.int32, device=dev)
        out["ep_count"] = torch.zeros(E, dtype=torch.int32, device=dev)
        out["margin"] = torch.full((E, k_max + 1), float("nan"), dtype=torch.float32, device=dev)
        out["gap"] = torch.full((E, k_max + 1), float("nan"), dtype=torch.float32, device=dev)
        out["rounds"] = torch.zeros(E, dtype=torch.int32, device=dev)
    if memory:
        out["memory"] = torch.empty((sum(n_vis), sel.shape.D), dtype=torch.float32, device=dev)
    o = sp_select_out(ptr(out["idx"]), int(k_cap), ptr(out["count"]), ptr(out.get("order")),
                      ptr(out.get("ep_count")), ptr(out.get("margin")), ptr(out.get("gap")),
                      ptr(out.get("rounds")), ptr(out.get("memory")), ptr(out["err"]))
    if no_alloc:
        _check(lib().sp_select_noalloc(sel.handle, C.byref(inp), C.byref(o), _stream(stream)), "sp_select_noalloc")
        out["k_cap"] = k_cap
        return out
    if ws is None:
        ws = workspace(lib().sp_select_workspace(sel.handle, C.byref(inp)), dev)
    if train is not None:
        out["score"] = torch.empty(sum(n_vis), dtype=torch.float32, device=dev)
        out["kbar"] = torch.empty(E, dtype=torch.float32, device=dev)
        ta = sp_train_args(float(train[0]), float(train[1]), ptr(out["score"]), ptr(out["kbar"]))
        _check(lib().sp_select_train(sel.handle, C.byref(inp), C.byref(o), C.byref(ta), ptr(ws), ws.numel(),
                                     _stream(stream)), "sp_select_train")
        out["k_cap"] = k_cap
        out["_ws"] = ws
        return out
    _check(lib().sp_select(sel.handle, C.byref(inp), C.byref(o), ptr(ws), ws.numel(), _stream(stream)), "sp_select")
    out["k_cap"] = k_cap
    out["_ws"] = ws
    return out


def sp_soft_topk(n_vis, *, score, kbar, tau, group_size=0, stream=None, alpha=None) -> Dict:
    """Eq. 8 per image (k = the batch mean of the images' soft counts); returns
    alpha [sum N_b] fp32 and k [1] fp32 (device tensors)."""
    torch = _torch()
    dev = score.device
    nv = _int_array(n_vis)
    if alpha is None:
        alpha = torch.empty(sum(n_vis), dtype=torch.float32, device=dev)
    k = torch.empty(1, dtype=torch.float32, device=dev)
    _check(lib().sp_soft_topk(len(n_vis), C.cast(nv, IP), int(group_size), ptr(score), ptr(kbar), float(tau),
                              ptr(alpha), ptr(k), _stream(stream)), "sp_soft_topk")
    return {"alpha": alpha, "k": k}


def sp_vp_gate(*, X, noise, alpha, out=None, stream=None):
    """Eq. 9 on bf16 rows: out = sqrt(alpha) X + sqrt(1 - alpha) noise."""
    torch = _torch()
    if out is None:
        out = torch.empty_like(X)
    rows, D = X.shape
    _check(lib().sp_vp_gate(int(rows), int(D), ptr(X), ptr(noise), ptr(alpha), ptr(out), _stream(stream)),
           "sp_vp_gate")
    return out


# ----------------------------------------------------------------------------- compaction

def sp_compact(n_vis, n_txt, *, X, text, idx, count, k_cap, projector_mode=False, index_mode=False, stream=None,
               out: Optional[Dict] = None) -> Dict:
    """Compaction into new zero-filled outputs, or into `out` (a dict a
    previous call returned for the same sizes) without touching it first.
    projector_mode: the kept visual rows go to out['vis_packed'] (with their
    packed rows in 'vis_row_map'); index_mode: no visual row is copied,
    out['vis_src'] holds the row of X each kept visual row comes from."""
    torch = _torch()
    dev = X.device
    keep: List = []
    nv, nt = _int_array(n_vis), _int_array(n_txt)
    keep += [nv, nt]
    W_vis, W_txt = X.shape[1], text.shape[1]
    T_cap = sp_packed_cap(n_vis, n_txt, k_cap)
    rows_cap = sum(min(n, k_cap) for n in n_vis)
    mode = "index" if index_mode else ("projector" if projector_mode else "direct")
    if out is None:
        out = {"packed": torch.zeros((max(T_cap, 1), W_txt), dtype=torch.bfloat16, device=dev),
               "cu_seqlens": torch.zeros(len(n_vis) + 1, dtype=torch.int32, device=dev),
               "pos": torch.full((max(T_cap, 1),), -1, dtype=torch.int32, device=dev),
               "err": torch.zeros(1, dtype=torch.int32, device=dev), "T_cap": T_cap, "mode": mode}
        if mode != "direct":
            out["vis_row_map"] = torch.full((max(rows_cap, 1),), -1, dtype=torch.int32, device=dev)
            out["vis_cu"] = torch.zeros(len(n_vis) + 1, dtype=torch.int32, device=dev)
            out["rows_cap"] = rows_cap
        if mode == "projector":
            out["vis_packed"] = torch.zeros((max(rows_cap, 1), W_vis), dtype=torch.bfloat16, device=dev)
        if mode == "index":
            out["vis_src"] = torch.full((max(rows_cap, 1),), -1, dtype=torch.int32, device=dev)
    elif out["T_cap"] != T_cap or out.get("mode") != mode or (mode != "direct" and out.get("rows_cap") != rows_cap):
        raise ValueError("sp_compact: `out` was made for other sizes or another mode")
    ci = sp_compact_in(len(n_vis), C.cast(nv, IP), C.cast(nt, IP), ptr(X), int(W_vis), ptr(text), int(W_txt),
                       ptr(idx), int(k_cap), ptr(count))
    co = sp_compact_out(ptr(out["packed"]), ptr(out["cu_seqlens"]), ptr(out["pos"]), ptr(out.get("vis_packed")),
                        ptr(out.get("vis_row_map")), ptr(out.get("vis_cu")), ptr(out["err"]), ptr(out.get("vis_src")))
    _check(lib().sp_compact(C.byref(ci), C.byref(co), _stream(stream)), "sp_compact")
    return out


# ----------------------------------------------------------------------------- model

class Model:
    """An LM (projector + decoder) handle plus its device weights."""

    def __init__(self, shape, layers: Sequence[Dict], head: Dict, device="cuda", max_pos=8192,
                 device_weights=None):
        torch = _torch()
        self.shape, self.device = shape, torch.device(device)
        self._keep: List = []
        w = sp_model_weights()

        def keep(t):
            self._keep.append(t)
            return ptr(t)

        if device_weights is not None:  # already on the device
            layers = device_weights["layers"]
            head = device_weights["head"]
        for l, L in enumerate(layers):
            w.wqkv[l] = keep(dev_bf16(L["Wqkv"], device))
            w.wo[l] = keep(dev_bf16(L["Wo"], device))
            w.wgu[l] = keep(dev_bf16(L["Wgu"], device))
            w.wdown[l] = keep(dev_bf16(L["Wdown"], device))
            w.attn_norm[l] = keep(dev_f32(L["attn_norm"], device))
            w.mlp_norm[l] = keep(dev_f32(L["mlp_norm"], device))
        w.final_norm = keep(dev_f32(head["final_norm"], device))
        if head.get("proj_W1") is not None:
            w.proj_w1 = keep(dev_bf16(head["proj_W1"], device))
        if head.get("proj_W2") is not None:
            w.proj_w2 = keep(dev_bf16(head["proj_W2"], device))
        cfg = sp_model_cfg(len(layers), shape.d, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn,
                           int(max_pos), float(shape.rope_theta), float(shape.rms_eps), PROJ[shape.proj_kind],
                           shape.proj_in, shape.proj_hidden,
                           (C.c_int * 3)(*[int(v) for v in getattr(shape, "mrope_section", (0, 0, 0))]))
        h = P()
        _check(lib().sp_model_create(C.byref(cfg), C.byref(w), C.byref(h)), "sp_model_create")
        self.handle = h
        self._w = w

    def close(self):
        if getattr(self, "handle", None):
            lib().sp_model_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def sp_project(model: Model, *, vis_row_map, vis_cu, packed, rows_cap, B, vis_packed=None, X=None, vis_src=None,
               stream=None, ws=None):
    """The projector on the kept rows: from vis_packed (projector-mode
    compaction), or gathered from X by vis_src (index-mode compaction)."""
    torch = _torch()
    err = torch.zeros(1, dtype=torch.int32, device=packed.device)
    io = sp_project_io(int(B), int(rows_cap), ptr(vis_packed), ptr(vis_row_map), ptr(vis_cu), ptr(packed), ptr(err),
                       ptr(X), int(X.shape[0]) if X is not None else 0, ptr(vis_src))
    if ws is None:
        ws = workspace(lib().sp_project_workspace(model.handle, int(rows_cap)), packed.device)
    _check(lib().sp_project(model.handle, C.byref(io), ptr(ws), ws.numel(), _stream(stream)), "sp_project")
    return err


def kv_cache(model: Model, B: int, S_cap: int, device=None):
    """A zeroed key / value cache [n_layers, 2, B, S_cap, n_kv_heads * head_dim] bf16."""
    torch = _torch()
    m = model.shape
    return torch.zeros((m.n_layers, 2, B, S_cap, m.n_kv_heads * m.head_dim), dtype=torch.bfloat16,
                       device=device or model.device)


def sp_prefill(model: Model, *, x, cu_seqlens, pos, B, T_cap, max_seqlen_cap, residual=None, stream=None,
               ws=None, hidden=None, kv=None, pos3=None):
    torch = _torch()
    dev = x.device
    if hidden is None:
        hidden = torch.zeros((max(T_cap, 1), model.shape.d), dtype=torch.float32, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    io = sp_prefill_io(int(B), int(T_cap), int(max_seqlen_cap), ptr(x), ptr(cu_seqlens), ptr(pos), ptr(hidden),
                       ptr(residual), ptr(err), ptr(kv), int(kv.shape[3]) if kv is not None else 0, ptr(pos3))
    if ws is None:
        ws = workspace(lib().sp_prefill_workspace(model.handle, int(T_cap), int(max_seqlen_cap)), dev)
    _check(lib().sp_prefill(model.handle, C.byref(io), ptr(ws), ws.numel(), _stream(stream)), "sp_prefill")
    return {"hidden": hidden, "err": err, "_ws": ws}


def sp_decode(model: Model, *, x, lens, kv, max_len_cap, stream=None, ws=None, hidden=None, rope_pos=None) -> Dict:
    """One generation step: x [B, d] bf16 new tokens, lens [B] int32 cached lengths
    (incremented on the device), kv the cache of kv_cache() / sp_prefill;
    rope_pos [B] int32 rotary positions (default lens), incremented with lens."""
    torch = _torch()
    dev = x.device
    B = int(x.shape[0])
    if hidden is None:
        hidden = torch.zeros((B, model.shape.d), dtype=torch.float32, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    io = sp_decode_io(B, ptr(x), ptr(lens), ptr(kv), int(kv.shape[3]), int(max_len_cap), ptr(hidden), ptr(err),
                      ptr(rope_pos))
    if ws is None:
        ws = workspace(lib().sp_decode_workspace(model.handle, B), dev)
    _check(lib().sp_decode(model.handle, C.byref(io), ptr(ws), ws.numel(), _stream(stream)), "sp_decode")
    return {"hidden": hidden, "err": err, "_ws": ws}


def sp_mrope_positions(n_vis, n_txt, grid_w, *, idx, count, k_cap, T_cap, stream=None, pos3=None, err=None):
    """(t, h, w) rotary positions [T_cap, 4] int32 of the packed, pruned batch."""
    torch = _torch()
    dev = idx.device
    if pos3 is None:
        pos3 = torch.zeros((max(int(T_cap), 1), 4), dtype=torch.int32, device=dev)
    if err is None:
        err = torch.zeros(1, dtype=torch.int32, device=dev)
    nv, nt, gw = _int_array(n_vis), _int_array(n_txt), _int_array(grid_w)
    _check(lib().sp_mrope_positions(len(n_vis), C.cast(nv, IP), C.cast(nt, IP), C.cast(gw, IP), ptr(idx), int(k_cap),
                                    ptr(count), ptr(pos3), int(T_cap), ptr(err), _stream(stream)),
           "sp_mrope_positions")
    return {"pos3": pos3, "err": err}


class Pipeline:
    """Pre-sized buffers for repeated sp_pipeline calls on one batch shape."""

    def __init__(self, sel: Selector, model: Model, n_vis, n_txt, *, group_size, g, k_max, k_cap=None):
        torch = _torch()
        self.sel, self.model = sel, model
        self.n_vis, self.n_txt = list(n_vis), list(n_txt)
        self.group_size, self.g, self.k_max = group_size, g, k_max
        self.k_cap = k_cap if k_cap is not None else k_cap_for(n_vis, group_size, k_max)
        self.B = len(n_vis)
        self.T_cap = sp_packed_cap(n_vis, n_txt, self.k_cap)
        dev = sel.device
        self._nv, self._nt = _int_array(n_vis), _int_array(n_txt)
        self.idx = torch.empty((self.B, self.k_cap), dtype=torch.int32, device=dev)
        self.count = torch.empty(self.B, dtype=torch.int32, device=dev)
        self.cu = torch.empty(self.B + 1, dtype=torch.int32, device=dev)
        self.hidden = torch.empty((max(self.T_cap, 1), model.shape.d), dtype=torch.float32, device=dev)
        self.err = torch.zeros(1, dtype=torch.int32, device=dev)
        io = self._io(None, None, None)
        self.ws = workspace(lib().sp_pipeline_workspace(sel.handle, model.handle, C.byref(io)), dev)
        self._host = None

    def _sel_in(self, X, E, bias):
        return sp_select_in(self.B, C.cast(self._nv, IP), C.cast(self._nt, IP), X, E, None, bias,
                            int(self.group_size), int(self.g), int(self.k_max))

    def _io(self, X, E, bias):
        return sp_pipeline_io(self._sel_in(ptr(X), ptr(E), ptr(bias)), int(self.k_cap), ptr(self.idx),
                              ptr(self.count), ptr(self.cu), ptr(self.hidden), ptr(self.err))

    def __call__(self, X, E_text, stop_bias, stream=None):
        """sp_pipeline on device inputs; results stay in self.idx / count / cu / hidden."""
        io = self._io(X, E_text, stop_bias)
        _check(lib().sp_pipeline(self.sel.handle, self.model.handle, C.byref(io), ptr(self.ws), self.ws.numel(),
                                 _stream(stream)), "sp_pipeline")

    def host(self, X_host, E_host, bias_host, out_idx, out_count, out_cu, out_hidden, stream=None):
        """sp_pipeline_host on (pinned) host tensors; outputs written to host tensors."""
        torch = _torch()
        io = sp_pipeline_host_io(self._sel_in(ptr(X_host), ptr(E_host), ptr(bias_host)), int(self.k_cap),
                                 ptr(out_idx), ptr(out_count), ptr(out_cu), ptr(out_hidden))
        if self._host is None:
            n = lib().sp_pipeline_host_workspace(self.sel.handle, self.model.handle, C.byref(io))
            self._host = workspace(n, self.sel.device)
        _check(lib().sp_pipeline_host(self.sel.handle, self.model.handle, C.byref(io), ptr(self._host),
                                      self._host.numel(), _stream(stream)), "sp_pipeline_host")


def sp_profile_begin(capacity: int = 1 << 16):
    _check(lib().sp_profile_begin(int(capacity)), "sp_profile_begin")


def sp_profile_end() -> Dict[str, Dict[str, float]]:
    n = len(KERNEL_KINDS)
    ms = (C.c_double * n)()
    la = (C.c_longlong * n)()
    fl = (C.c_double * n)()
    by = (C.c_double * n)()
    _check(lib().sp_profile_end(ms, la, fl, by), "sp_profile_end")
    return {k: {"ms": ms[i], "launches": int(la[i]), "flops": fl[i], "bytes": by[i]}
            for i, k in enumerate(KERNEL_KINDS)}


def sp_wait_probe(*, flag, limit_us: int, complete: bool, out, err=None, stream=None):
    """The bounded-wait self-test: out[0] / out[1] = 1 if the mbarrier / flag
    wait completed, 0 if it ran out after limit_us (SP_DEVERR_TIMEOUT in err)."""
    _check(lib().sp_wait_probe(ptr(flag), int(limit_us), 1 if complete else 0, ptr(out), ptr(err), _stream(stream)),
           "sp_wait_probe")


def sp_device_error_status(word: int) -> int:
    return lib().sp_device_error_status(int(word))
