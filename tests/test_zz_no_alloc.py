"""snapkv_score_noalloc: the SnapKV score for callers that cannot allocate
device memory (a serving process whose allocator already owns all of HBM, a
plugin that only receives its input and output buffers, a path that must not
pay cudaMalloc's synchronisation).  It keeps its scratch in the library's own
static device array instead of a caller workspace.

Checked through the C ABI against snapkv_score (the workspace version) on two
calls in a row with different shapes, so that whatever the first call left in
the shared array cannot leak into the second.  This file is collected last.
"""

import ctypes

import numpy as np
import pytest
import torch

from paper_2607_13205_gb300 import inputs as I
from paper_2607_13205_gb300 import rolekv as R
from tests.gpu_helpers import assert_scores_close, lib_batch, oracle_batch

pytestmark = pytest.mark.gpu

DEV = "cuda"


def _case(w, seed, pool_k):
    roles = I.workload_roles(w, seed)
    K, _ = I.make_kv(w, roles, seed, device=DEV, with_v=False)
    qw = I.make_q_window(w, seed, device=DEV)
    batch = lib_batch(w, DEV)
    # reference: the existing entry point with a caller workspace
    ref = torch.empty(batch.score_shape(), dtype=torch.float32, device=DEV)
    ref_pre = torch.empty_like(ref)
    R.snapkv_score(batch, qw, K, w.W, pool_k, ref, scores_prepool=ref_pre)
    # no-allocation entry point
    out = torch.full_like(ref, -1.0)
    out_pre = torch.full_like(ref, -1.0) if pool_k > 1 else None
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.snapkv_score_noalloc(batch, qw, K, w.W, pool_k, out, scores_prepool=out_pre, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ob = oracle_batch(w)
    got, want = out.cpu().numpy(), ref.cpu().numpy()
    for u in range(ob.n_units):
        assert_scores_close(ob.score_view(got, u), ob.score_view(want, u).astype(np.float64),
                            f"unit {u}")
        if out_pre is not None:
            assert_scores_close(ob.score_view(out_pre.cpu().numpy(), u),
                                ob.score_view(ref_pre.cpu().numpy(), u).astype(np.float64),
                                f"unit {u} pre-pool")


def test_noalloc_matches_workspace_version_twice():
    # first call: a dense batch with two row tiles and several key chunks
    w1 = I.WORKLOADS["long"].scaled(L=2, b=2, Hq=8, Hkv=2, n=9000)
    _case(w1, seed=21, pool_k=7)
    # second call, right after: a smaller varlen batch with an empty and a
    # short sequence, no pooling
    w2 = I.WORKLOADS["ragged"].scaled(L=1, b=4, Hq=14, Hkv=2, n=3000, seqlens=(3000, 0, 20, 1500))
    _case(w2, seed=22, pool_k=1)


def test_noalloc_rejects_oversized_batches():
    # 64 layers x 64 sequences x 8 KV heads at 16384 tokens needs more scratch
    # than the static array holds; the call must refuse before touching the GPU
    b = R.BatchDesc(64, 64, 32, 8, 128, 16384, None, None)
    t = R.Tensor(16, 0, 0, 0, 128)
    f = ctypes.c_void_p(256)
    rc = R.lib().snapkv_score_noalloc(ctypes.byref(b), t, t, 32, 1, 0.0, None, f, None, None, None)
    assert rc == R.ERR_UNSUPPORTED
    assert b"scratch" in R.lib().rolekv_last_error()
    # pooling without a pre-pool output buffer is refused too
    small = R.BatchDesc(1, 1, 8, 2, 128, 1000, None, None)
    rc = R.lib().snapkv_score_noalloc(ctypes.byref(small), t, t, 32, 7, 0.0, None, f, None, None, None)
    assert rc == R.ERR_INVALID_ARG
