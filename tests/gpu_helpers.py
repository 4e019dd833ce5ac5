"""Shared helpers of the GPU parity tests: run the library on seeded inputs and
compare with the fp64 oracle under the stated tolerances."""

from __future__ import annotations

import numpy as np
import torch

from oracle import rolekv_oracle as O
from paper_2607_13205_gb300 import inputs as I
from paper_2607_13205_gb300 import rolekv as R

# Scores: fp32 accumulation from bf16 inputs agrees with the fp64 oracle to
# 1e-3 relative (the tolerance the method's statement fixes); the tiny absolute
# floor only admits values below fp32's exp2 range.
SCORE_RTOL = 1e-3
SCORE_ATOL = 1e-20


def assert_scores_close(got: np.ndarray, ref: np.ndarray, what: str = ""):
    got = np.asarray(got, dtype=np.float64)
    err = np.abs(got - ref)
    bound = SCORE_RTOL * np.abs(ref) + SCORE_ATOL
    bad = np.nonzero(err > bound)[0]
    assert bad.size == 0, (f"{what}: {bad.size} scores off; first t={bad[0]} got={got[bad[0]]!r} "
                           f"ref={ref[bad[0]]!r} rel={err[bad[0]] / max(abs(ref[bad[0]]), 1e-300):.3g}")


def oracle_batch(w: I.Workload, kept_extra: int = 0) -> O.Batch:
    return O.Batch(w.L, w.b, w.Hq, w.Hkv, w.d, w.n, seqlens=list(w.seqlens) if w.varlen else None,
                   kept_extra=kept_extra)


def lib_batch(w: I.Workload, device, kept_extra: int = 0) -> R.Batch:
    return R.Batch(w.L, w.b, w.Hq, w.Hkv, w.d, w.n, seqlens=list(w.seqlens) if w.varlen else None,
                   device=device, kept_extra=kept_extra)


def check_index_sets(ob: O.Batch, u: int, got_idx: np.ndarray, ref_scores: np.ndarray, roles_np,
                     n_roles, alpha, key_role, alpha_key, budget, policy=O.POLICY_ROLE_QUOTA,
                     ban_mask=0):
    """Kept sets from fp32 GPU scores vs the oracle's fp64 scores: same size and
    per-bucket counts, and any position in one set but not the other has an
    oracle score within 1e-3 relative of its bucket's k-th threshold."""
    ref = O.select_batch(ob, {u: ref_scores}, roles_np, n_roles, alpha, key_role, alpha_key, budget,
                         policy, ban_mask)[u][0]
    got = np.asarray(got_idx)
    assert got.shape == ref.shape
    assert np.array_equal(got < 0, ref < 0), "padding differs"
    g = set(int(x) for x in got if x >= 0)
    r = set(int(x) for x in ref if x >= 0)
    assert len(g) == len(r)
    assert np.all(np.diff(got[got >= 0]) > 0), "kept positions must ascend"
    _, s, _ = ob.unit(u)
    roles = np.asarray(ob.roles(roles_np, s)).astype(np.int64)
    buckets = O.bucket_of_tokens(roles, policy, ban_mask)
    al = [float(np.float32(a)) for a in alpha[:n_roles]]
    if 0 <= key_role < n_roles:
        al[key_role] = float(np.float32(alpha_key))
    q = O.role_quotas([int((roles == x).sum()) for x in range(n_roles)], al, budget, roles.size,
                      policy, ban_mask)
    for t in g ^ r:
        bk = buckets[t]
        assert bk >= 0
        members = np.nonzero(buckets == bk)[0]
        thr = np.sort(ref_scores[members])[::-1][q[bk] - 1]
        assert abs(ref_scores[t] - thr) <= SCORE_RTOL * abs(thr), (
            f"unit {u}: position {t} differs and its score {ref_scores[t]} is not near the "
            f"threshold {thr}")
    for bk in range(n_roles):
        mem = buckets == bk
        assert sum(1 for t in g if mem[t]) == sum(1 for t in r if mem[t])


def window_lse_oracle(w: I.Workload, ob: O.Batch, qb, kb) -> np.ndarray:
    """Natural-log softmax normaliser of every SnapKV window row over its
    causal keys, fp64 on the host from the bf16 inputs, stored as fp32
    [L][b][Hq][W] (rows i >= W_eff left at 0): the LSE a prefill attention
    hands over."""
    lse = np.zeros((w.L, w.b, w.Hq, w.W), dtype=np.float32)
    scale = 1.0 / np.sqrt(w.d)
    for u in range(ob.n_units):
        l, s, h = ob.unit(u)
        k = O.bf16_to_f64(ob.kv_rows(kb, u))
        n = k.shape[0]
        if n == 0:
            continue
        w_eff = min(w.W, n)
        for g in range(w.G):
            q = O.bf16_to_f64(qb[l, s, h * w.G + g, :w_eff])
            logits = scale * (q @ k.T)
            for i in range(w_eff):
                row = logits[i, :n - w_eff + i + 1]
                m = row.max()
                lse[l, s, h * w.G + g, i] = m + np.log(np.exp(row - m).sum())
    return lse


def prefill_lse_oracle(w: I.Workload, ob: O.Batch, qb, kb) -> np.ndarray:
    """Natural-log softmax normaliser of every causal prefill query row, fp64
    on the host from the bf16 inputs, stored as fp32 in the layout h2o_score
    takes: dense [L][b][Hq][n_max], varlen [L][Hq][T]."""
    shape = (w.L, w.Hq, ob.T) if w.varlen else (w.L, w.b, w.Hq, w.n)
    lse = np.zeros(shape, dtype=np.float32)
    scale = 1.0 / np.sqrt(w.d)
    for u in range(ob.n_units):
        l, s, h = ob.unit(u)
        k = O.bf16_to_f64(ob.kv_rows(kb, u))
        n = k.shape[0]
        if n == 0:
            continue
        q = O.bf16_to_f64(ob.q_rows(qb, u))           # (G, n, d)
        causal = np.arange(n)[None, :] <= np.arange(n)[:, None]
        for g in range(w.G):
            logits = np.where(causal, scale * (q[g] @ k.T), -np.inf)
            m = logits.max(axis=1, keepdims=True)
            row_lse = (m + np.log(np.exp(logits - m).sum(axis=1, keepdims=True)))[:, 0]
            if w.varlen:
                c0 = int(ob.cu[s])
                lse[l, h * w.G + g, c0:c0 + n] = row_lse
            else:
                lse[l, s, h * w.G + g, :n] = row_lse
    return lse
