"""Seeded sweep over shapes: random small configurations (head dim, GQA group,
window, pool width, length mix with empty and very short sequences, budget,
policy, recency floor, kept-row widening), each taken through score -> select -> compact ->
decode on the GPU and compared with the fp64 oracle: scores within 1e-3
relative, selection and compaction bit-exact on the kernel's own scores,
decode within the decode tolerance; half of them also through the H2O score
and the Quest page bound."""

import numpy as np
import pytest
import torch

from oracle import rolekv_oracle as O
from paper_2607_13205_gb300 import inputs as I
from paper_2607_13205_gb300 import rolekv as R
from tests.gpu_helpers import assert_scores_close, lib_batch, oracle_batch

pytestmark = pytest.mark.gpu

DEV = "cuda"
N_CASES = 24


def _config(seed):
    g = np.random.default_rng(np.random.SeedSequence([seed, 0xF022]))
    d = int(g.choice([64, 128]))
    G = int(g.choice([1, 2, 4, 7, 8]))
    W = int(g.choice([w for w in (8, 16, 32, 64) if w * G <= 256]))
    Hkv = int(g.integers(1, 3))
    b = int(g.integers(1, 4))
    n = int(g.choice([1, 2, 5, 31, 129, 777, 1500, 2600]))
    varlen = bool(g.random() < 0.5)
    seqlens = None
    if varlen:
        seqlens = tuple(int(x) for x in g.choice([0, 1, 3, 64, 200, 1000, n], size=b))
        n = max(max(seqlens), 1)
        seqlens = tuple(min(x, n) for x in seqlens)
    w = I.WORKLOADS["tiny"].scaled(L=1, b=b, Hq=G * Hkv, Hkv=Hkv, d=d, n=n, W=W,
                                   pool_k=int(g.choice([1, 3, 5, 7, 15])), seqlens=seqlens)
    B = float(g.choice([0.01, 0.05, 0.1, 0.3, 0.5, 1.0]))
    policy = int(g.integers(0, 5))
    keep_last = int(g.choice([0, 0, 4, 40]))
    akey = float(g.choice([0.0, 0.02]))
    ban = int(1 << I.ROLE_KEY) if g.random() < 0.2 else 0
    extra = int(g.choice([0, 0, 0, 2]))
    if policy == R.POLICY_CEIL:
        extra = I.N_ROLES - 1 + extra
    return w, B, policy, keep_last, akey, ban, extra


@pytest.mark.parametrize("seed", list(range(N_CASES)))
def test_random_configuration_end_to_end(seed):
    w, B, policy, keep_last, akey, ban, extra = _config(seed)
    roles_np = I.workload_roles(w, seed)
    K, V = I.make_kv(w, roles_np, seed, device=DEV)
    qw = I.make_q_window(w, seed, device=DEV)
    batch = lib_batch(w, DEV, kept_extra=extra)
    ob = oracle_batch(w, kept_extra=extra)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)

    scores = torch.full(batch.score_shape(), -1.0, dtype=torch.float32, device=DEV)
    R.snapkv_score(batch, qw, K, w.W, w.pool_k, scores, status=status)
    params = R.select_params(B, I.PAPER_ALPHA, alpha_key=akey, key_role=I.ROLE_KEY, policy=policy,
                             ban_mask=ban, keep_last=keep_last)
    keep = torch.full(batch.kept_shape(B), -7, dtype=torch.int32, device=DEV)
    per_role = torch.full((batch.n_units, I.N_ROLES), -1, dtype=torch.int32, device=DEV)
    R.role_alloc_select(batch, scores, torch.as_tensor(roles_np, device=DEV), params, keep,
                        kept_per_role=per_role, status=status)
    kc = torch.empty(R.compact_shape(batch, B), dtype=torch.bfloat16, device=DEV)
    vc = torch.empty_like(kc)
    R.kv_compact(batch, K, V, keep, B, kc, vc, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0, f"status {int(status.item())}"

    # scores
    ref = O.snapkv_batch(ob, I.bf16_bits(qw), I.bf16_bits(K), w.W, w.pool_k)
    got = scores.cpu().numpy()
    for u, (_, pooled) in ref.items():
        assert_scores_close(ob.score_view(got, u), pooled, f"seed {seed} unit {u}")

    # selection on the kernel's scores, and compaction of the kept rows
    sel = O.select_batch(ob, {u: ob.score_view(got, u).astype(np.float64) for u in range(ob.n_units)},
                         roles_np, I.N_ROLES, I.PAPER_ALPHA, I.ROLE_KEY, akey, B, policy, ban,
                         keep_last=keep_last)
    cu = ob.kept_offsets(B)
    kp, pr = keep.cpu().numpy(), per_role.cpu().numpy()
    kb, vb = I.bf16_bits(K), I.bf16_bits(V)
    kcb, vcb = I.bf16_bits(kc), I.bf16_bits(vc)

    def rows(arr, u):
        l, s, h = ob.unit(u)
        return arr[l, h, cu[s]:cu[s + 1]] if ob.varlen else arr.reshape((ob.n_units, -1) + arr.shape[4:])[u]

    for u, (idx, per) in sel.items():
        assert np.array_equal(rows(kp, u), idx), f"seed {seed} unit {u}: kept set"
        assert list(pr[u]) == per, f"seed {seed} unit {u}: per-role counts"
        assert np.array_equal(rows(kcb, u), O.compact_unit(ob.kv_rows(kb, u), idx)), f"seed {seed} unit {u}: K"
        assert np.array_equal(rows(vcb, u), O.compact_unit(ob.kv_rows(vb, u), idx)), f"seed {seed} unit {u}: V"

    # one decode step through the compacted cache
    qd = I.make_q_decode(w, seed, device=DEV)
    out = torch.full((w.L, w.b, w.Hq, w.d), float("nan"), dtype=torch.float32, device=DEV)
    R.decode_attention(batch, qd, kc, vc, keep, B, out, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    o = out.cpu().numpy()
    qdb = I.bf16_bits(qd)
    vmax = float(V.float().abs().max()) if V.numel() else 1.0
    for u in range(ob.n_units):
        l, s, h = ob.unit(u)
        idx = rows(kp, u)
        r = O.decode_attention(O.bf16_to_f64(qdb[l, s, h * w.G:(h + 1) * w.G]),
                               O.bf16_to_f64(rows(kcb, u)), O.bf16_to_f64(rows(vcb, u)), idx >= 0,
                               1.0 / np.sqrt(w.d))
        got_o = o[l, s, h * w.G:(h + 1) * w.G].astype(np.float64)
        assert np.all(np.abs(got_o - r) <= 1e-3 * np.abs(r) + 1e-4 * vmax), f"seed {seed} unit {u}: decode"


@pytest.mark.parametrize("seed", list(range(0, N_CASES, 2)))
def test_random_configuration_h2o_and_quest(seed):
    """The same seeded configurations through the H2O score (every causal
    query, n kept at most 1500 for the oracle) and the Quest page bound."""
    w, B, policy, keep_last, akey, ban, _ = _config(seed)
    if w.n > 1500:
        w = w.scaled(n=1500, seqlens=None if w.seqlens is None else tuple(min(x, 1500) for x in w.seqlens))
    roles_np = I.workload_roles(w, seed)
    K, _ = I.make_kv(w, roles_np, seed, device=DEV, with_v=False)
    Q = I.make_q_full(w, seed, device=DEV)
    qw = I.make_q_window(w, seed, device=DEV)
    batch = lib_batch(w, DEV)
    ob = oracle_batch(w)
    scores = torch.full(batch.score_shape(), -1.0, dtype=torch.float32, device=DEV)
    R.h2o_score(batch, Q, K, scores)
    torch.cuda.synchronize()
    ref = O.h2o_batch(ob, I.bf16_bits(Q), I.bf16_bits(K))
    got = scores.cpu().numpy()
    for u, s in ref.items():
        assert_scores_close(ob.score_view(got, u), s, f"seed {seed} unit {u} h2o")

    page = int(np.random.default_rng(seed).choice([1, 4, 16, 33]))
    qs = torch.full(batch.score_shape(), float("nan"), dtype=torch.float32, device=DEV)
    R.quest_score(batch, qw, K, w.W, page, qs)
    torch.cuda.synchronize()
    qb, kb = I.bf16_bits(qw), I.bf16_bits(K)
    qref = O.quest_batch(ob, qb, kb, w.W, page)
    qgot = qs.cpu().numpy()
    for u, r in qref.items():
        g = ob.score_view(qgot, u).astype(np.float64)
        l, s, h = ob.unit(u)
        k = O.bf16_to_f64(ob.kv_rows(kb, u))
        n = k.shape[0]
        if n == 0:
            continue
        w_eff = min(w.W, n)
        qbar = np.abs(O.bf16_to_f64(qb[l, s, h * w.G:(h + 1) * w.G, :w_eff]).reshape(-1, w.d).mean(axis=0))
        tol = 1e-5 * qbar.sum() * np.abs(k).max() + 1e-4 * np.abs(r)
        assert np.all(np.abs(g - r) <= tol), f"seed {seed} unit {u} quest"
