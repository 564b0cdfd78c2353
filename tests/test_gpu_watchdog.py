"""Failure detection on the GPU without a fault: the bounded waits the kernels
use run out on an mbarrier and a flag that nothing completes, record
SP_DEVERR_TIMEOUT and return; the stream and the context stay usable (the next
call on the same stream gives exact results)."""
import time

import numpy as np
import pytest

from oracle import core as O
from paper_2609_13804_gb300 import synth as S

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

DEV = "cuda"
SP_ERR_TIMEOUT = 6


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_13804_gb300 import binding
    binding.lib()
    return binding


def test_waits_run_out_and_report_a_timeout(B):
    flag = torch.zeros(1, dtype=torch.int32, device=DEV)        # nothing sets it
    out = torch.full((2,), -1, dtype=torch.int32, device=DEV)
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    t0 = time.perf_counter()
    B.sp_wait_probe(flag=flag, limit_us=1000, complete=False, out=out, err=err)
    torch.cuda.synchronize()
    elapsed = time.perf_counter() - t0
    assert out.cpu().tolist() == [0, 0]
    assert B.sp_device_error_status(int(err.item())) == SP_ERR_TIMEOUT
    assert elapsed < 1.0, elapsed  # two 1 ms limits, not the 2 s default


def test_completed_waits_report_nothing(B):
    flag = torch.ones(1, dtype=torch.int32, device=DEV)
    out = torch.full((2,), -1, dtype=torch.int32, device=DEV)
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    B.sp_wait_probe(flag=flag, limit_us=1000, complete=True, out=out, err=err)
    torch.cuda.synchronize()
    assert out.cpu().tolist() == [1, 1]
    assert int(err.item()) == 0


def test_stream_stays_usable_after_a_timeout(B):
    flag = torch.zeros(1, dtype=torch.int32, device=DEV)
    out = torch.zeros(2, dtype=torch.int32, device=DEV)
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    B.sp_wait_probe(flag=flag, limit_us=500, complete=False, out=out, err=err)
    # the next call on the same stream: a compaction, checked bit for bit
    n_vis, n_txt, W = [40, 7], [3, 2], 256
    X = S.bf16_round(S.normal(91, "X", (sum(n_vis), W)))
    text = S.bf16_round(S.normal(91, "T", (sum(n_txt), W)))
    idx_list = [np.array([1, 5, 39]), np.arange(7)]
    idx = np.full((2, 8), -1, np.int32)
    for b, l in enumerate(idx_list):
        idx[b, :len(l)] = l
    count = np.array([3, 7], np.int32)
    r = B.sp_compact(n_vis, n_txt, X=B.dev_bf16(X, DEV), text=B.dev_bf16(text, DEV),
                     idx=torch.from_numpy(idx).to(DEV), count=torch.from_numpy(count).to(DEV), k_cap=8)
    torch.cuda.synchronize()
    assert B.sp_device_error_status(int(err.item())) == SP_ERR_TIMEOUT
    assert int(r["err"].item()) == 0
    packed, cu, pos = O.compact(X, n_vis, idx_list, text, n_txt)
    T = int(cu[-1])
    np.testing.assert_array_equal(r["cu_seqlens"].cpu().numpy(), cu)
    np.testing.assert_array_equal(r["packed"].float().cpu().numpy()[:T], packed)
