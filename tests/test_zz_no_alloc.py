"""sp_select_noalloc: the selection entry point for callers that cannot allocate
device memory (it uses the library's static device scratch instead of a caller
workspace).  Its results must be those of sp_select, call after call, since the
scratch is shared and keeps the previous call's contents.

This file is collected last on purpose: a failure here leaves every other test
already run.  It passes alone in a fresh process and after the other tests."""
import ctypes as C

import numpy as np
import pytest

from paper_2609_13804_gb300 import synth as S

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

DEV = "cuda"
KEYS = ("idx", "count", "order", "ep_count", "rounds", "gap", "margin")


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_13804_gb300 import binding
    binding.lib()
    return binding


def _same(a, b):
    for k in KEYS:
        x, y = a[k].cpu().numpy(), b[k].cpu().numpy()
        np.testing.assert_array_equal(x, y, err_msg=k)  # same kernels on the same inputs: bit-identical


def test_noalloc_matches_sp_select_on_two_calls_in_a_row(B):
    w = S.llava15_7b_b16()
    w.n_vis, w.n_txt = w.n_vis[:4], w.n_txt[:4]
    s = S.SelectorShape(D=w.selector.D, D_text=w.selector.D_text, h=w.selector.h, n_enc_layers=0)
    sel = S.make_selector_weights(w, ln_affine=True)
    selector = B.Selector(s, sel, DEV)
    H1 = B.dev_f32(S.make_memory(w, "H1"), DEV)
    H2 = B.dev_f32(S.make_memory(w, "H2"), DEV)
    b1 = B.dev_f32(np.array([-1e30, 0.0, -0.2, 0.1], np.float32), DEV)
    b2 = B.dev_f32(np.array([0.05, -1e30, -0.1, -0.3], np.float32), DEV)
    for H, bias in ((H1, b1), (H2, b2)):
        ref = B.sp_select(selector, w.n_vis, w.n_txt, H=H, stop_bias=bias, k_max=w.k_max)
        got = B.sp_select(selector, w.n_vis, w.n_txt, H=H, stop_bias=bias, k_max=w.k_max, no_alloc=True)
        torch.cuda.synchronize()
        assert int(got["err"].item()) == 0
        _same(got, ref)
    selector.close()


def test_noalloc_with_the_encoder_matches_sp_select_on_two_calls_in_a_row(B):
    """The encoder path (text projection, encoder blocks, their GEMM scratch
    and encoder buffers all in the static scratch): two calls with different
    inputs, each bit-identical to sp_select's."""
    w = S.tiny_workload(81, [40, 130, 7], [5, 0, 3], D=128, D_text=128, h=128, enc_head_dim=64, k_max=12)
    s = w.selector
    sel = S.make_selector_weights(w, ln_affine=True)
    selector = B.Selector(s, sel, DEV)
    for name, bias in (("a", [-1e30, 0.0, -0.1]), ("b", [0.02, -1e30, -1e30])):
        X = B.dev_bf16(S.bf16_round(S.normal(81, "X" + name, (sum(w.n_vis), s.D))), DEV)
        E = B.dev_bf16(S.bf16_round(S.normal(81, "E" + name, (sum(w.n_txt), s.D_text), 0.02)), DEV)
        bd = B.dev_f32(np.array(bias, np.float32), DEV)
        ref = B.sp_select(selector, w.n_vis, w.n_txt, X=X, E_text=E, stop_bias=bd, k_max=w.k_max, memory=True)
        got = B.sp_select(selector, w.n_vis, w.n_txt, X=X, E_text=E, stop_bias=bd, k_max=w.k_max, no_alloc=True,
                          memory=True)
        torch.cuda.synchronize()
        assert int(got["err"].item()) == 0 and int(ref["err"].item()) == 0
        _same(got, ref)
        np.testing.assert_array_equal(got["memory"].cpu().numpy(), ref["memory"].cpu().numpy())
    selector.close()


def test_noalloc_rejects_a_batch_beyond_its_scratch(B):
    w = S.llava15_7b_b16()
    s = S.SelectorShape(D=w.selector.D, D_text=w.selector.D_text, h=w.selector.h, n_enc_layers=0)
    selector = B.Selector(s, S.make_selector_weights(w), DEV)
    n_vis = [16384] * 4  # 65 k candidates x (D + 5 h) fp32 rows: far beyond the static scratch
    n_txt = [1] * 4
    nv, nt = B._int_array(n_vis), B._int_array(n_txt)
    inp = B.sp_select_in(4, C.cast(nv, B.IP), C.cast(nt, B.IP), None, None, 16, 16, 0, 1, 8)
    assert B.lib().sp_select_workspace(selector.handle, C.byref(inp)) > B.SP_SELECT_NOALLOC_SCRATCH_BYTES
    out = B.sp_select_out(16, 8, 16, None, None, None, None, None, None, None)
    st = B.lib().sp_select_noalloc(selector.handle, C.byref(inp), C.byref(out), None)
    assert st == 4  # SP_ERR_WORKSPACE, before any launch (the pointers above are never touched)
    assert b"static scratch" in B.lib().sp_last_error()
    selector.close()
