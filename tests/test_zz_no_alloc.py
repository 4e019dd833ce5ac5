"""snapkv_score_noalloc: the SnapKV score for callers that cannot allocate
device memory (a serving process whose allocator already owns all of HBM, a
plugin that only receives its input and output buffers, a path that must not
pay cudaMalloc's synchronisation).  It keeps its scratch in the library's own
static device array instead of a caller workspace.

Checked through the C ABI against the fp64 oracle and against snapkv_score
(the workspace version), on calls in a row with different shapes, so that
whatever one call left in the shared array cannot leak into the next.  The
calls cover both kernels this entry point runs (two passes, or one pass with
caller-supplied window normalisers) and both head dimensions.  The host-side
rejections (a batch too large for the array, pooling without a pre-pool
buffer) are checked on the CPU, in tests/test_abi.py.  This file is
collected last.
"""

import numpy as np
import pytest
import torch

from oracle import rolekv_oracle as O
from paper_2607_13205_gb300 import inputs as I
from paper_2607_13205_gb300 import rolekv as R
from tests.gpu_helpers import assert_scores_close, lib_batch, oracle_batch, window_lse_oracle

pytestmark = pytest.mark.gpu

DEV = "cuda"


def _case(w, seed, pool_k, supply_lse=False):
    roles = I.workload_roles(w, seed)
    K, _ = I.make_kv(w, roles, seed, device=DEV, with_v=False)
    qw = I.make_q_window(w, seed, device=DEV)
    batch = lib_batch(w, DEV)
    ob = oracle_batch(w)
    qb, kb = I.bf16_bits(qw), I.bf16_bits(K)
    lse = torch.as_tensor(window_lse_oracle(w, ob, qb, kb), device=DEV) if supply_lse else None
    # reference: the existing entry point with a caller workspace
    ref = torch.empty(batch.score_shape(), dtype=torch.float32, device=DEV)
    ref_pre = torch.empty_like(ref)
    R.snapkv_score(batch, qw, K, w.W, pool_k, ref, scores_prepool=ref_pre, lse_win=lse)
    # no-allocation entry point
    out = torch.full_like(ref, -1.0)
    out_pre = torch.full_like(ref, -1.0) if pool_k > 1 else None
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.snapkv_score_noalloc(batch, qw, K, w.W, pool_k, out, scores_prepool=out_pre, lse_win=lse,
                           status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    oracle = O.snapkv_batch(ob, qb, kb, w.W, pool_k)
    got, want = out.cpu().numpy(), ref.cpu().numpy()
    got_pre = out_pre.cpu().numpy() if out_pre is not None else None
    for u, (rpre, rpool) in oracle.items():
        g = ob.score_view(got, u)
        assert_scores_close(g, rpool, f"unit {u} against the oracle")
        assert_scores_close(g, ob.score_view(want, u).astype(np.float64), f"unit {u} against snapkv_score")
        if got_pre is not None:
            assert_scores_close(ob.score_view(got_pre, u), rpre, f"unit {u} pre-pool against the oracle")


def test_noalloc_matches_oracle_and_workspace_version_in_a_row():
    # first call: a dense batch with two row tiles and several key chunks
    w1 = I.WORKLOADS["long"].scaled(L=2, b=2, Hq=8, Hkv=2, n=9000)
    _case(w1, seed=21, pool_k=7)
    # second call, right after: a smaller varlen batch with an empty and a
    # short sequence, no pooling
    w2 = I.WORKLOADS["ragged"].scaled(L=1, b=4, Hq=14, Hkv=2, n=3000, seqlens=(3000, 0, 20, 1500))
    _case(w2, seed=22, pool_k=1)
    # third: d = 64 with the window normalisers supplied (one pass over K)
    w3 = I.WORKLOADS["tiny"].scaled(L=1, b=2, n=2500)
    _case(w3, seed=23, pool_k=5, supply_lse=True)


def test_noalloc_empty_batch_needs_no_output():
    # every sequence empty: nothing to write, so no output buffer is needed
    # (the same as snapkv_score)
    w = I.WORKLOADS["ragged"].scaled(L=1, b=2, Hq=8, Hkv=2, n=64, seqlens=(0, 0))
    batch = lib_batch(w, DEV)
    qw = torch.zeros((1, 2, 8, w.W, w.d), dtype=torch.bfloat16, device=DEV)
    k = torch.zeros((1, 1, 2, w.d), dtype=torch.bfloat16, device=DEV)
    R.snapkv_score_noalloc(batch, qw, k, w.W, 7, None, scores_prepool=None)
