"""GPU parity at the full sizes of the five benchmark configurations, in the
launch configuration bench.py times (snapkv_score with pre-pool output, the
selector with the pool fused, kv_compact; h2o_score for the H2O config).

Sampled units are compared with the fp64 oracle (scores to 1e-3 relative, kept
sets up to ties within 1e-3 of the bucket threshold, compaction bit-exact);
every unit is checked for the properties that hold at any size: each window
row is a distribution (pre-pool mass totals W_eff*G, H2O mass n*G), exactly
ceil(B n) slots with ascending in-range indices, per-role counts consistent
with the roles, no KEY token kept when alpha_KEY = 0."""

import gc

import numpy as np
import pytest
import torch

from oracle import rolekv_oracle as O
from paper_2607_13205_gb300 import inputs as I
from paper_2607_13205_gb300 import rolekv as R
from tests.gpu_helpers import assert_scores_close, check_index_sets, lib_batch, oracle_batch

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(autouse=True)
def _free_memory():
    yield
    gc.collect()
    torch.cuda.empty_cache()


class UnitView:
    """One (layer, sequence, KV head) of a batch copied to the host as a
    single-unit dense oracle batch."""

    def __init__(self, w, ob, u, K, V, roles_np, qw=None, Q=None):
        self.u = u
        l, s, h = ob.unit(u)
        n = ob.seqlens[s]
        G = w.G
        if ob.varlen:
            c0, c1 = int(ob.cu[s]), int(ob.cu[s + 1])
            krows, vrows = K[l, c0:c1, h], V[l, c0:c1, h]
            qfull = None if Q is None else Q[l, c0:c1, h * G:(h + 1) * G].transpose(0, 1)
        else:
            krows, vrows = K[l, s, h, :n], V[l, s, h, :n]
            qfull = None if Q is None else Q[l, s, h * G:(h + 1) * G, :n]
        self.k = I.bf16_bits(krows)[None, None, None]
        self.v = I.bf16_bits(vrows)[None, None, None]
        self.qw = None if qw is None else I.bf16_bits(qw[l, s, h * G:(h + 1) * G])[None, None]
        self.q = None if qfull is None else I.bf16_bits(qfull)[None, None]
        self.roles = np.asarray(ob.roles(roles_np, s))[None, :]
        self.ob = O.Batch(1, 1, G, 1, w.d, n)


def _unit_rows(ob, arr, u, kept_offsets):
    l, s, h = ob.unit(u)
    if ob.varlen:
        return arr[l, h, kept_offsets[s]:kept_offsets[s + 1]]
    return arr.reshape((ob.n_units, -1) + arr.shape[4:])[u]


def _run_snapkv_path(w, B, seed=0, alpha_key=0.0):
    roles_np = I.workload_roles(w, seed)
    K, V = I.make_kv(w, roles_np, seed, device=DEV)
    qw = I.make_q_window(w, seed, device=DEV)
    roles = torch.as_tensor(roles_np, device=DEV)
    batch = lib_batch(w, DEV)
    params = R.select_params(B, I.PAPER_ALPHA, alpha_key, I.ROLE_KEY)
    pre = torch.empty(batch.score_shape(), dtype=torch.float32, device=DEV)
    keep = torch.empty(batch.kept_shape(B), dtype=torch.int32, device=DEV)
    k_out = torch.empty(R.compact_shape(batch, B), dtype=torch.bfloat16, device=DEV)
    v_out = torch.empty_like(k_out)
    per_role = torch.empty((batch.n_units, I.N_ROLES), dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.snapkv_score(batch, qw, K, w.W, 1, pre, status=status)
    R.role_alloc_select(batch, pre, roles, params, keep, pool_k=w.pool_k, kept_per_role=per_role,
                        status=status)
    R.kv_compact(batch, K, V, keep, B, k_out, v_out, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return dict(roles=roles_np, K=K, V=V, qw=qw, scores=pre.cpu().numpy(), keep=keep.cpu().numpy(),
                k_out=k_out, v_out=v_out, per_role=per_role.cpu().numpy())


def _check_all_units(w, B, ob, r, alpha_key, mass_per_unit):
    kept_off = ob.kept_offsets(B)
    for u in range(ob.n_units):
        _, s, _ = ob.unit(u)
        n = ob.seqlens[s]
        sc = ob.score_view(r["scores"], u).astype(np.float64)
        if n:
            total = mass_per_unit(n)
            assert abs(sc.sum() - total) <= 1e-3 * total, (u, sc.sum(), total)
        row = _unit_rows(ob, r["keep"], u, kept_off)
        assert row.size == (O.kept_count(n, B) if n else 0)
        kept = row[row >= 0]
        assert np.all(np.diff(kept) > 0) and (kept.size == 0 or (kept[0] >= 0 and kept[-1] < n))
        roles_u = np.asarray(ob.roles(r["roles"], s))
        counts = np.bincount(roles_u[kept], minlength=I.N_ROLES)[:I.N_ROLES]
        assert list(counts) == list(r["per_role"][u])
        if alpha_key == 0.0:
            assert counts[I.ROLE_KEY] == 0


def _check_sampled_snapkv(w, B, ob, units, r, alpha_key):
    kept_off = ob.kept_offsets(B)
    ko_all, vo_all = I.bf16_bits(r["k_out"]), I.bf16_bits(r["v_out"])
    for u in units:
        v = UnitView(w, ob, u, r["K"], r["V"], r["roles"], qw=r["qw"])
        pre, pooled = O.snapkv_batch(v.ob, v.qw, v.k, w.W, w.pool_k)[0]
        assert_scores_close(ob.score_view(r["scores"], u), pre, f"{w.name} unit {u} pre-pool")
        row = _unit_rows(ob, r["keep"], u, kept_off)
        check_index_sets(v.ob, 0, row, pooled, v.roles, I.N_ROLES, I.PAPER_ALPHA, I.ROLE_KEY,
                         alpha_key, B)
        assert np.array_equal(_unit_rows(ob, ko_all, u, kept_off), O.compact_unit(v.k[0, 0, 0], row))
        assert np.array_equal(_unit_rows(ob, vo_all, u, kept_off), O.compact_unit(v.v[0, 0, 0], row))


def _check_ceil_select(w, B, r, units):
    """The literal ceiling split (rows N_ROLES - 1 slots wider) on the
    kernel's own scores: bit-exact against the oracle on the sampled units;
    on every unit the row is ascending, -1 padded, and keeps between
    ceil(B n) and ceil(B n) + 3 tokens, counted per role."""
    extra = I.N_ROLES - 1
    batch = lib_batch(w, DEV, kept_extra=extra)
    ob = oracle_batch(w, kept_extra=extra)
    pre = torch.as_tensor(r["scores"], device=DEV)
    params = R.select_params(B, I.PAPER_ALPHA, 0.0, I.ROLE_KEY, policy=R.POLICY_CEIL)
    keep = torch.full(batch.kept_shape(B), -7, dtype=torch.int32, device=DEV)
    per_role = torch.empty((batch.n_units, I.N_ROLES), dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.role_alloc_select(batch, pre, torch.as_tensor(r["roles"], device=DEV), params, keep,
                        pool_k=w.pool_k, kept_per_role=per_role, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    keep_np, pr = keep.cpu().numpy(), per_role.cpu().numpy()
    kept_off = ob.kept_offsets(B)
    for u in range(ob.n_units):
        n = ob.seqlens[ob.unit(u)[1]]
        row = _unit_rows(ob, keep_np, u, kept_off)
        assert row.size == ob.kept_rows(n, B)
        kept = row[row >= 0]
        assert np.all(row[kept.size:] == -1) and np.all(np.diff(kept) > 0)
        K = O.kept_count(n, B)
        assert K <= kept.size <= K + extra and int(pr[u].sum()) == kept.size, (u, kept.size, K)
    for u in units:
        sc = O.maxpool1d(ob.score_view(r["scores"], u).astype(np.float64), w.pool_k)
        idx, per = O.select_batch(ob, {u: sc}, r["roles"], I.N_ROLES, I.PAPER_ALPHA, I.ROLE_KEY, 0.0,
                                  B, O.POLICY_CEIL)[u]
        assert np.array_equal(_unit_rows(ob, keep_np, u, kept_off), idx), f"ceil unit {u}"
        assert list(pr[u]) == per


def _check_slack_select(w, B, r, units, alpha_key=0.02):
    """The SLACK fill (first-round quotas, the slack of saturated buckets to
    the best-scoring unkept tokens of eligible roles) on the kernel's own
    scores: every unit keeps exactly min(ceil(B n), eligible) tokens in an
    ascending row counted per role; bit-exact against the oracle on the
    sampled units."""
    batch = lib_batch(w, DEV)
    ob = oracle_batch(w)
    pre = torch.as_tensor(r["scores"], device=DEV)
    params = R.select_params(B, I.PAPER_ALPHA, alpha_key, I.ROLE_KEY, policy=R.POLICY_SLACK)
    keep = torch.full(batch.kept_shape(B), -7, dtype=torch.int32, device=DEV)
    per_role = torch.empty((batch.n_units, I.N_ROLES), dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.role_alloc_select(batch, pre, torch.as_tensor(r["roles"], device=DEV), params, keep,
                        pool_k=w.pool_k, kept_per_role=per_role, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    keep_np, pr = keep.cpu().numpy(), per_role.cpu().numpy()
    kept_off = ob.kept_offsets(B)
    alpha = list(I.PAPER_ALPHA)
    alpha[I.ROLE_KEY] = alpha_key
    for u in range(ob.n_units):
        s = ob.unit(u)[1]
        n = ob.seqlens[s]
        row = _unit_rows(ob, keep_np, u, kept_off)
        kept = row[row >= 0]
        assert np.all(row[kept.size:] == -1) and np.all(np.diff(kept) > 0)
        counts = np.bincount(np.asarray(ob.roles(r["roles"], s)), minlength=I.N_ROLES)[:I.N_ROLES]
        eligible = int(sum(c for c, a in zip(counts, alpha) if a > 0))
        assert kept.size == min(O.kept_count(n, B), eligible), (u, kept.size)
        assert int(pr[u].sum()) == kept.size
    for u in units:
        sc = O.maxpool1d(ob.score_view(r["scores"], u).astype(np.float64), w.pool_k)
        idx, per = O.select_batch(ob, {u: sc}, r["roles"], I.N_ROLES, I.PAPER_ALPHA, I.ROLE_KEY,
                                  alpha_key, B, O.POLICY_SLACK)[u]
        assert np.array_equal(_unit_rows(ob, keep_np, u, kept_off), idx), f"slack unit {u}"
        assert list(pr[u]) == per


def test_long_context_full_size():
    """L=32, b=4, N=32768, 32/8 heads, d=128, W=64, pool 7, B=0.10 (~17 GB K/V)."""
    w = I.WORKLOADS["long"]
    B = w.budgets[0]
    r = _run_snapkv_path(w, B)
    ob = oracle_batch(w)
    _check_all_units(w, B, ob, r, 0.0, lambda n: min(w.W, n) * w.G)
    _check_sampled_snapkv(w, B, ob, [0, 517, ob.n_units - 1], r, 0.0)
    _check_ceil_select(w, B, r, [0, 517, ob.n_units - 1])
    _check_slack_select(w, B, r, [3, 600, ob.n_units - 1])
    _check_one_call(w, B, ob, r, [5, 700, ob.n_units - 2])


def _check_one_call(w, B, ob, r, units):
    """rolekv_compress (score, select with the pool fused, compaction in one
    call) on the same inputs: kept indices, per-role counts and compressed
    K/V bit-exact against the three separate calls, and against the oracle on
    the sampled units."""
    batch = lib_batch(w, DEV)
    params = R.select_params(B, I.PAPER_ALPHA, 0.0, I.ROLE_KEY)
    keep = torch.full(batch.kept_shape(B), -7, dtype=torch.int32, device=DEV)
    k_out = torch.empty(R.compact_shape(batch, B), dtype=torch.bfloat16, device=DEV)
    v_out = torch.empty_like(k_out)
    per_role = torch.empty((batch.n_units, I.N_ROLES), dtype=torch.int32, device=DEV)
    ws = R.workspace(R.OP_COMPRESS, batch, w.W, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.rolekv_compress(batch, r["qw"], r["K"], r["V"], w.W, w.pool_k, torch.as_tensor(r["roles"], device=DEV),
                      params, keep, k_out, v_out, ws, kept_per_role=per_role, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert np.array_equal(keep.cpu().numpy(), r["keep"])
    assert np.array_equal(per_role.cpu().numpy(), r["per_role"])
    assert torch.equal(k_out, r["k_out"]) and torch.equal(v_out, r["v_out"])
    r1 = dict(r, keep=keep.cpu().numpy(), k_out=k_out, v_out=v_out)
    _check_sampled_snapkv(w, B, ob, units, r1, 0.0)


@pytest.mark.parametrize("B", I.WORKLOADS["llama8b"].budgets)
def test_llama8b_full_size_every_budget(B):
    """L=32, b=1, N=8192, 32/8 heads, d=128, W=32, pool 7, five budgets
    (alpha_KEY = 0.02, the cross-model default, at two of them)."""
    w = I.WORKLOADS["llama8b"]
    akey = 0.02 if B in (0.10, 0.30) else 0.0
    r = _run_snapkv_path(w, B, seed=1, alpha_key=akey)
    ob = oracle_batch(w)
    _check_all_units(w, B, ob, r, akey, lambda n: min(w.W, n) * w.G)
    _check_sampled_snapkv(w, B, ob, [3, 130, ob.n_units - 1], r, akey)


def test_ragged_full_size():
    """64 sequences of 1024..16384 tokens, 28 layers, 28/4 heads, W=32, B=0.10,
    packed varlen K/V."""
    w = I.WORKLOADS["ragged"]
    B = w.budgets[0]
    r = _run_snapkv_path(w, B, seed=2)
    ob = oracle_batch(w)
    _check_all_units(w, B, ob, r, 0.0, lambda n: min(w.W, n) * w.G)
    lens = list(w.seqlens)
    s_short, s_long = int(np.argmin(lens)), int(np.argmax(lens))
    units = [s_short * w.Hkv, s_long * w.Hkv + 3, (w.L - 1) * w.b * w.Hkv + 17 * w.Hkv + 1]
    _check_sampled_snapkv(w, B, ob, units, r, 0.0)


def test_h2o_full_size():
    """H2O accumulated mass over all 8192 causal queries, b=2, 32/8 heads,
    d=128, L=32 (the config leaves L open), then selection at B=0.05 (no pool)
    and compaction."""
    w = I.WORKLOADS["h2o"]
    B = w.budgets[0]
    roles_np = I.workload_roles(w, 3)
    K, V = I.make_kv(w, roles_np, 3, device=DEV)
    Q = I.make_q_full(w, 3, device=DEV)
    batch = lib_batch(w, DEV)
    scores = torch.empty(batch.score_shape(), dtype=torch.float32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.h2o_score(batch, Q, K, scores, status=status)
    params = R.select_params(B, I.PAPER_ALPHA, 0.0, I.ROLE_KEY)
    keep = torch.empty(batch.kept_shape(B), dtype=torch.int32, device=DEV)
    per_role = torch.empty((batch.n_units, I.N_ROLES), dtype=torch.int32, device=DEV)
    R.role_alloc_select(batch, scores, torch.as_tensor(roles_np, device=DEV), params, keep,
                        kept_per_role=per_role, status=status)
    k_out = torch.empty(R.compact_shape(batch, B), dtype=torch.bfloat16, device=DEV)
    v_out = torch.empty_like(k_out)
    R.kv_compact(batch, K, V, keep, B, k_out, v_out, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ob = oracle_batch(w)
    r = dict(roles=roles_np, scores=scores.cpu().numpy(), keep=keep.cpu().numpy(),
             per_role=per_role.cpu().numpy())
    _check_all_units(w, B, ob, r, 0.0, lambda n: n * w.G)
    kept_off = ob.kept_offsets(B)
    ko_all = I.bf16_bits(k_out)
    for u in (261,):
        v = UnitView(w, ob, u, K, V, roles_np, Q=Q)
        ref = O.h2o_batch(v.ob, v.q, v.k)[0]
        assert_scores_close(ob.score_view(r["scores"], u), ref, f"h2o unit {u}")
        row = _unit_rows(ob, r["keep"], u, kept_off)
        check_index_sets(v.ob, 0, row, ref, v.roles, I.N_ROLES, I.PAPER_ALPHA, I.ROLE_KEY, 0.0, B)
        assert np.array_equal(_unit_rows(ob, ko_all, u, kept_off), O.compact_unit(v.k[0, 0, 0], row))


def test_quest_long_full_size():
    """Quest one-shot analogue on the long config (page 16, mean query of the
    64-row window), then page top-k (GLOBAL, B=0.10) and compaction."""
    w = I.WORKLOADS["long"]
    B, page = w.budgets[0], 16
    roles_np = I.workload_roles(w, 4)
    K, V = I.make_kv(w, roles_np, 4, device=DEV)
    qw = I.make_q_window(w, 4, device=DEV)
    batch = lib_batch(w, DEV)
    scores = torch.empty(batch.score_shape(), dtype=torch.float32, device=DEV)
    R.quest_score(batch, qw, K, w.W, page, scores)
    params = R.select_params(B, I.PAPER_ALPHA, 0.0, I.ROLE_KEY, policy=R.POLICY_GLOBAL)
    keep = torch.empty(batch.kept_shape(B), dtype=torch.int32, device=DEV)
    R.role_alloc_select(batch, scores, torch.as_tensor(roles_np, device=DEV), params, keep)
    k_out = torch.empty(R.compact_shape(batch, B), dtype=torch.bfloat16, device=DEV)
    v_out = torch.empty_like(k_out)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.kv_compact(batch, K, V, keep, B, k_out, v_out, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ob = oracle_batch(w)
    sc = scores.cpu().numpy().reshape(ob.n_units, -1)
    assert np.all(np.isfinite(sc))
    assert np.all(sc.reshape(ob.n_units, -1, page) == sc.reshape(ob.n_units, -1, page)[:, :, :1])
    kp = keep.cpu().numpy().reshape(ob.n_units, -1)
    Ks = O.kept_count(w.n, B)
    assert kp.shape[1] == Ks and np.all(np.diff(kp, axis=1) > 0)
    ko = I.bf16_bits(k_out).reshape(ob.n_units, Ks, -1)
    for u in (0, 611, ob.n_units - 1):
        v = UnitView(w, ob, u, K, V, roles_np, qw=qw)
        ref = O.quest_score(O.bf16_to_f64(v.qw[0, 0]), O.bf16_to_f64(v.k[0, 0, 0]), w.W, page)
        scale = np.abs(O.bf16_to_f64(v.qw[0, 0]).reshape(-1, w.d)[:w.G * w.W].mean(axis=0)).sum()
        tol = 1e-5 * scale * np.abs(O.bf16_to_f64(v.k[0, 0, 0])).max() + 1e-4 * np.abs(ref)
        assert np.all(np.abs(sc[u] - ref) <= tol)
        check_index_sets(v.ob, 0, kp[u], ref, v.roles, I.N_ROLES, I.PAPER_ALPHA, I.ROLE_KEY, 0.0, B,
                         policy=O.POLICY_GLOBAL)
        # on the kernel's own page bounds the selection is bit-exact (these
        # narrow-range, page-constant keys take the selector's extra digit
        # rounds and its tie ranking)
        exact = O.select_batch(ob, {u: sc[u].astype(np.float64)}, roles_np, I.N_ROLES, I.PAPER_ALPHA,
                               I.ROLE_KEY, 0.0, B, O.POLICY_GLOBAL)
        assert np.array_equal(kp[u], exact[u][0])
        assert np.array_equal(ko[u], O.compact_unit(v.k[0, 0, 0], kp[u]))
