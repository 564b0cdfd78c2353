"""Host-side checks of the C ABI: the library loads without a GPU, exports every
symbol include/stepprune.h declares, and its host arithmetic / argument checks
behave.  No kernel is launched."""
import ctypes as C
import os
import re

import pytest

from paper_2609_13804_gb300 import binding as b

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    if not os.path.exists(b.LIB_PATH):
        from paper_2609_13804_gb300 import build
        build.build()
    return b.lib()


def declared_symbols():
    with open(os.path.join(ROOT, "include", "stepprune.h")) as f:
        src = f.read()
    return sorted(set(re.findall(r"^SP_API [^(]*?\b(sp_[a-z0-9_]+)\(", src, flags=re.M)))


def test_header_and_binding_agree():
    assert declared_symbols() == sorted(b.EXPORTS)


def test_library_exports_every_declared_symbol(L):
    for name in declared_symbols():
        assert hasattr(L, name), name
    assert L.sp_abi_version() == 1


def test_struct_sizes_match_header_layout():
    # pointer arrays sized by the header limits; a mismatch shifts every later field
    assert C.sizeof(b.sp_selector_weights) == 8 * (3 + 8 * b.SP_MAX_ENC_LAYERS + 13 + 1)
    assert C.sizeof(b.sp_selector_cfg) == 4 * 9
    assert C.sizeof(b.sp_dec_layer_weights) == 8 * 16
    assert C.sizeof(b.sp_model_weights) == 8 * (6 * b.SP_MAX_LM_LAYERS + 3)
    assert C.sizeof(b.sp_select_in) == 4 + 4 + 8 * 6 + 4 * 3 + 4
    assert C.sizeof(b.sp_select_out) == 8 + 8 + 8 * 8


def test_prefill_and_decode_io_layout():
    assert C.sizeof(b.sp_prefill_io) == 4 * 3 + 4 + 8 * 6 + 8 + 4 + 4 + 8
    assert C.sizeof(b.sp_decode_io) == 4 + 4 + 8 * 3 + 4 * 2 + 8 * 2 + 8
    assert C.sizeof(b.sp_model_cfg) == 4 * 15


def test_decode_argument_checks_fail_before_any_launch(L):
    assert L.sp_decode(None, None, None, 0, None) == 1
    assert L.sp_decode_workspace(None, 4) == 0


def test_host_arithmetic(L):
    assert b.sp_num_episodes([576] * 16, 0) == 16
    assert b.sp_num_episodes([2880] * 8, 576) == 40
    assert b.sp_num_episodes([1025, 1024, 1], 1024) == 4
    assert b.sp_packed_cap([576, 100], [48, 3], 192) == 192 + 48 + 100 + 3
    assert b.k_cap_for([2880], 576, 128) == 640
    assert b.k_cap_for([1100], 1024, 256) == 256 + 76
    assert L.sp_num_episodes(0, None, 0) == -1
    assert L.sp_packed_cap(1, b._int_array([0]), b._int_array([1]), 4) == -1


def test_device_error_word_mapping(L):
    assert L.sp_device_error_status(0) == 0
    assert L.sp_device_error_status(1) == 6  # SP_ERR_TIMEOUT
    assert L.sp_device_error_status(2) == 8  # SP_ERR_DEVICE
    assert b"0x2" in L.sp_last_error()


def test_argument_checks_fail_before_any_launch(L):
    assert L.sp_compact(None, None, None) == 1
    nv, nt = b._int_array([4]), b._int_array([2])
    ci = b.sp_compact_in(1, C.cast(nv, b.IP), C.cast(nt, b.IP), None, 8, None, 8, None, 4, None)
    co = b.sp_compact_out()
    assert L.sp_compact(C.byref(ci), C.byref(co), None) == 1  # X / idx / outputs missing
    ci = b.sp_compact_in(1, C.cast(nv, b.IP), C.cast(nt, b.IP), 16, 12, 32, 8, 48, 4, 64)
    co = b.sp_compact_out(80, 96, 112, None, None, None, None)
    assert L.sp_compact(C.byref(ci), C.byref(co), None) == 2  # W_vis not a multiple of 8
    ci = b.sp_compact_in(1, C.cast(nv, b.IP), C.cast(nt, b.IP), 8, 8, 32, 8, 48, 4, 64)
    assert L.sp_compact(C.byref(ci), C.byref(co), None) == 3  # X misaligned
    ci = b.sp_compact_in(1, C.cast(nv, b.IP), C.cast(nt, b.IP), 16, 8, 32, 8, 48, 4, 64)
    co = b.sp_compact_out(80, 96, 112, 128, 144, 160, None, 176)
    assert L.sp_compact(C.byref(ci), C.byref(co), None) == 1  # vis_src and vis_packed together
    co = b.sp_compact_out(80, 96, 112, None, None, None, None, 176)
    assert L.sp_compact(C.byref(ci), C.byref(co), None) == 1  # index mode without vis_row_map / vis_cu
    assert L.sp_profile_end(None, None, None, None) == 1       # not started


def test_compact_and_project_io_layout():
    assert C.sizeof(b.sp_compact_out) == 8 * 8
    assert C.sizeof(b.sp_project_io) == 4 * 2 + 8 * 5 + 8 + 4 + 4 + 8


def test_create_without_a_gpu_reports_instead_of_crashing(L):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    cfg = b.sp_selector_cfg(1024, 1024, 256, 2, 64, 4096, 1e-5, 1.0)
    w = b.sp_selector_weights()
    h = b.P()
    st = L.sp_selector_create(C.byref(cfg), C.byref(w), C.byref(h))
    assert st in (5, 7)  # SP_ERR_CUDA / SP_ERR_UNSUPPORTED
    assert not h.value


def test_training_pathway_layout_and_argument_checks(L):
    assert C.sizeof(b.sp_train_args) == 4 + 4 + 8 + 8
    assert L.sp_select_train(None, None, None, None, None, 0, None) == 1   # no train arguments
    nv = b._int_array([4, 3])
    ok = C.c_void_p(256)  # never dereferenced: every call below fails on the host first
    assert L.sp_soft_topk(0, C.cast(nv, b.IP), 0, ok, ok, 0.1, ok, None, None) == 1       # B = 0
    assert L.sp_soft_topk(2, C.cast(nv, b.IP), 0, None, ok, 0.1, ok, None, None) == 1     # no scores
    assert L.sp_soft_topk(2, C.cast(nv, b.IP), 0, ok, ok, 0.0, ok, None, None) == 1       # tau = 0
    assert L.sp_soft_topk(2, C.cast(nv, b.IP), -1, ok, ok, 0.1, ok, None, None) == 2      # bad group size
    assert L.sp_vp_gate(4, 12, ok, ok, ok, ok, None) == 2                                  # D not a multiple of 8
    assert L.sp_vp_gate(0, 16, None, None, None, None, None) == 0                          # nothing to do
    assert L.sp_vp_gate(4, 16, None, ok, ok, ok, None) == 1
    assert L.sp_vp_gate(4, 16, C.c_void_p(264), ok, ok, ok, None) == 3                     # X misaligned


def test_mrope_argument_checks(L):
    nv, nt, gw = b._int_array([16, 9]), b._int_array([2, 3]), b._int_array([4, 3])
    ok = C.c_void_p(256)
    args = lambda g, kc, p: (2, C.cast(nv, b.IP), C.cast(nt, b.IP), C.cast(g, b.IP), ok, kc, ok, p, 64, None, None)  # noqa: E731
    assert L.sp_mrope_positions(*args(gw, 0, ok)) == 2                      # k_cap 0
    assert L.sp_mrope_positions(*args(b._int_array([4, 10]), 8, ok)) == 2  # grid wider than the image
    assert L.sp_mrope_positions(*args(gw, 8, None)) == 1
    assert L.sp_mrope_positions(*args(gw, 8, C.c_void_p(260))) == 3         # pos3 misaligned


def test_wait_probe_argument_checks_fail_before_any_launch(L):
    one = C.c_int(0)
    assert L.sp_wait_probe(None, 1000, 0, C.byref(one), None, None) == 1      # SP_ERR_INVALID_ARG: no flag
    assert L.sp_wait_probe(C.byref(one), 0, 0, C.byref(one), None, None) == 2  # SP_ERR_SHAPE: limit 0
    assert L.sp_wait_probe(C.byref(one), 2000001, 0, C.byref(one), None, None) == 2
    assert L.sp_device_error_status(0x1) == 6   # SP_DEVERR_TIMEOUT -> SP_ERR_TIMEOUT
