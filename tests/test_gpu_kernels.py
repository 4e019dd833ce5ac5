"""GPU parity: every entry point of librolekv against the fp64 oracle, through
the C ABI, on seeded synthetic inputs (sizes that span several tiles, a
ragged tail, varlen batches with empty and short sequences)."""

import numpy as np
import pytest
import torch

from oracle import rolekv_oracle as O
from paper_2607_13205_gb300 import inputs as I
from paper_2607_13205_gb300 import rolekv as R
from tests.gpu_helpers import (assert_scores_close, check_index_sets, lib_batch, oracle_batch,
                               prefill_lse_oracle, window_lse_oracle)

pytestmark = pytest.mark.gpu

DEV = "cuda"


def _w(name="tiny", **kw):
    return I.WORKLOADS[name].scaled(**kw)


SNAPKV_CASES = {
    "tiny_d64": _w("tiny"),
    "ragged_tail_g4w32": _w("llama8b", L=2, b=2, Hq=8, Hkv=2, n=1000),
    "two_row_tiles_w64_multichunk": _w("long", L=1, b=1, Hq=8, Hkv=2, n=8500),
    "g7_224_rows": _w("ragged", L=1, b=2, Hq=14, Hkv=2, n=2100, seqlens=None),
    "varlen_short_empty": _w("ragged", L=2, b=5, Hq=8, Hkv=2, n=2049, seqlens=(1000, 17, 0, 300, 2049)),
    "varlen_g7": _w("ragged", L=1, b=3, Hq=14, Hkv=2, n=1500, seqlens=(1500, 31, 640)),
}


def _snapkv_inputs(w, seed=0):
    roles = I.workload_roles(w, seed)
    K, V = I.make_kv(w, roles, seed, device=DEV)
    qw = I.make_q_window(w, seed, device=DEV)
    return roles, K, V, qw


@pytest.mark.parametrize("case", list(SNAPKV_CASES))
def test_snapkv_score_matches_oracle(case):
    w = SNAPKV_CASES[case]
    roles, K, V, qw = _snapkv_inputs(w)
    batch = lib_batch(w, DEV)
    scores = torch.full(batch.score_shape(), -1.0, dtype=torch.float32, device=DEV)
    pre = torch.full_like(scores, -1.0)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.snapkv_score(batch, qw, K, w.W, w.pool_k, scores, scores_prepool=pre, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ob = oracle_batch(w)
    ref = O.snapkv_batch(ob, I.bf16_bits(qw), I.bf16_bits(K), w.W, w.pool_k)
    got, gpre = scores.cpu().numpy(), pre.cpu().numpy()
    for u, (rpre, rpool) in ref.items():
        assert_scores_close(ob.score_view(gpre, u), rpre, f"{case} unit {u} pre-pool")
        assert_scores_close(ob.score_view(got, u), rpool, f"{case} unit {u} pooled")
        n = rpre.size
        if n:
            assert abs(ob.score_view(gpre, u).astype(np.float64).sum() - min(w.W, n) * w.G) < 1e-3 * min(w.W, n) * w.G


@pytest.mark.parametrize("pool_k", [5, 11])
@pytest.mark.parametrize("case", ["ragged_tail_g4w32", "varlen_short_empty"])
def test_snapkv_score_pool_widths(case, pool_k):
    """The standalone max-pool at the paper's other swept widths (Section 4),
    dense and varlen (pools never cross a sequence boundary)."""
    w = SNAPKV_CASES[case]
    roles, K, V, qw = _snapkv_inputs(w, seed=5)
    batch = lib_batch(w, DEV)
    scores = torch.full(batch.score_shape(), -1.0, dtype=torch.float32, device=DEV)
    R.snapkv_score(batch, qw, K, w.W, pool_k, scores)
    torch.cuda.synchronize()
    ob = oracle_batch(w)
    ref = O.snapkv_batch(ob, I.bf16_bits(qw), I.bf16_bits(K), w.W, pool_k)
    got = scores.cpu().numpy()
    for u, (_, rpool) in ref.items():
        assert_scores_close(ob.score_view(got, u), rpool, f"{case} pool {pool_k} unit {u}")


@pytest.mark.parametrize("scale", [0.004, 0.5])
@pytest.mark.parametrize("case", ["two_row_tiles_w64_multichunk", "varlen_g7"])
def test_snapkv_and_h2o_with_explicit_scale(case, scale):
    """A softmax scale other than 1/sqrt(d), from nearly flat (0.004) to
    sharply peaked (0.5): both score kernels against the oracle at that scale
    (the row normalisers enter pass 2 divided by scale * log2 e)."""
    w = SNAPKV_CASES[case]
    roles, K, V, qw = _snapkv_inputs(w, seed=4)
    batch = lib_batch(w, DEV)
    ob = oracle_batch(w)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    pre = torch.full(batch.score_shape(), -1.0, dtype=torch.float32, device=DEV)
    R.snapkv_score(batch, qw, K, w.W, 1, pre, scale=scale, status=status)
    ww = w if w.n <= 2100 else w.scaled(n=2100)
    Kh = K if ww is w else K[:, :, :, :ww.n].contiguous()
    bh = batch if ww is w else lib_batch(ww, DEV)
    obh = ob if ww is w else oracle_batch(ww)
    Q = I.make_q_full(ww, 4, device=DEV)
    hs = torch.full(bh.score_shape(), -1.0, dtype=torch.float32, device=DEV)
    R.h2o_score(bh, Q, Kh, hs, scale=scale, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ref = O.snapkv_batch(ob, I.bf16_bits(qw), I.bf16_bits(K), w.W, 1, scale=scale)
    got = pre.cpu().numpy()
    for u, (rpre, _) in ref.items():
        assert_scores_close(ob.score_view(got, u), rpre, f"{case} scale {scale} unit {u} snapkv")
    href = O.h2o_batch(obh, I.bf16_bits(Q), I.bf16_bits(Kh), scale=scale)
    hgot = hs.cpu().numpy()
    for u, r in href.items():
        assert_scores_close(obh.score_view(hgot, u), r, f"{case} scale {scale} unit {u} h2o")


@pytest.mark.parametrize("case", ["varlen_short_empty", "two_row_tiles_w64_multichunk", "varlen_g7"])
def test_snapkv_with_supplied_lse(case):
    """Single pass with the window rows' normalisers given (natural log, fp32,
    from the oracle's fp64 logits)."""
    w = SNAPKV_CASES[case]
    roles, K, V, qw = _snapkv_inputs(w, seed=3)
    ob = oracle_batch(w)
    kb, qb = I.bf16_bits(K), I.bf16_bits(qw)
    lse = window_lse_oracle(w, ob, qb, kb)
    batch = lib_batch(w, DEV)
    scores = torch.empty(batch.score_shape(), dtype=torch.float32, device=DEV)
    R.snapkv_score(batch, qw, K, w.W, w.pool_k, scores, lse_win=torch.as_tensor(lse, device=DEV))
    torch.cuda.synchronize()
    ref = O.snapkv_batch(ob, qb, kb, w.W, w.pool_k)
    got = scores.cpu().numpy()
    for u, (_, rpool) in ref.items():
        assert_scores_close(ob.score_view(got, u), rpool, f"{case} unit {u}")


H2O_CASES = {
    "dense_g4_ragged": _w("h2o", L=1, b=2, Hq=8, Hkv=2, n=700),
    "dense_g7": _w("h2o", L=1, b=1, Hq=14, Hkv=2, n=450),
    "varlen": _w("h2o", L=2, b=4, Hq=8, Hkv=2, n=300, seqlens=(300, 129, 0, 64)),
    "d64": _w("h2o", L=1, b=1, Hq=8, Hkv=2, d=64, n=520),
}


@pytest.mark.parametrize("case", list(H2O_CASES))
def test_h2o_score_matches_oracle(case):
    w = H2O_CASES[case]
    roles = I.workload_roles(w, 1)
    K, _ = I.make_kv(w, roles, 1, device=DEV, with_v=False)
    Q = I.make_q_full(w, 1, device=DEV)
    batch = lib_batch(w, DEV)
    scores = torch.full(batch.score_shape(), -1.0, dtype=torch.float32, device=DEV)
    R.h2o_score(batch, Q, K, scores)
    torch.cuda.synchronize()
    ob = oracle_batch(w)
    ref = O.h2o_batch(ob, I.bf16_bits(Q), I.bf16_bits(K))
    got = scores.cpu().numpy()
    for u, s in ref.items():
        assert_scores_close(ob.score_view(got, u), s, f"{case} unit {u}")
        if s.size:
            assert abs(ob.score_view(got, u).astype(np.float64).sum() - s.size * w.G) < 1e-3 * s.size * w.G


@pytest.mark.parametrize("case", list(H2O_CASES))
def test_h2o_score_with_supplied_lse(case):
    """One pass over K with every query row's natural-log normaliser given
    (fp32, from the oracle's fp64 logits; dense [L][b][Hq][n], varlen
    [L][Hq][T]): against the oracle, and against the two-pass score."""
    w = H2O_CASES[case]
    roles = I.workload_roles(w, 2)
    K, _ = I.make_kv(w, roles, 2, device=DEV, with_v=False)
    Q = I.make_q_full(w, 2, device=DEV)
    batch = lib_batch(w, DEV)
    ob = oracle_batch(w)
    qb, kb = I.bf16_bits(Q), I.bf16_bits(K)
    lse = torch.as_tensor(prefill_lse_oracle(w, ob, qb, kb), device=DEV)
    one = torch.full(batch.score_shape(), -1.0, dtype=torch.float32, device=DEV)
    two = torch.full_like(one, -1.0)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.h2o_score(batch, Q, K, one, lse=lse, status=status)
    R.h2o_score(batch, Q, K, two, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ref = O.h2o_batch(ob, qb, kb)
    g1, g2 = one.cpu().numpy(), two.cpu().numpy()
    for u, s in ref.items():
        assert_scores_close(ob.score_view(g1, u), s, f"{case} unit {u} one pass")
        assert_scores_close(ob.score_view(g1, u), ob.score_view(g2, u).astype(np.float64),
                            f"{case} unit {u} one pass against two")


# -------------------------------------------------------------------- quest

QUEST_CASES = {
    "tiny_d64_page16": (_w("tiny"), 16),
    "g4_page16_ragged_tail": (_w("llama8b", L=1, b=2, Hq=8, Hkv=2, n=3001), 16),
    "page1_is_dot": (_w("llama8b", L=1, b=1, Hq=8, Hkv=2, n=700), 1),
    "page64_w64": (_w("long", L=1, b=1, Hq=8, Hkv=2, n=5000), 64),
    "page5_g7": (_w("ragged", L=1, b=2, Hq=14, Hkv=2, n=2100, seqlens=None), 5),
    "varlen_short_empty": (SNAPKV_CASES["varlen_short_empty"], 16),
}


def _quest_tol(ob, qb, kb, u, W, G):
    """|qbar|_1 max|k|: the scale of the bound's rounding error."""
    l, s, h = ob.unit(u)
    k = O.bf16_to_f64(ob.kv_rows(kb, u))
    if k.shape[0] == 0:
        return 0.0
    q = O.bf16_to_f64(qb[l, s, h * G:(h + 1) * G, :min(W, k.shape[0])]).reshape(-1, k.shape[1])
    return float(np.abs(q.mean(axis=0)).sum() * np.abs(k).max())


@pytest.mark.parametrize("case", list(QUEST_CASES))
def test_quest_score_matches_oracle(case):
    w, page = QUEST_CASES[case]
    roles_np, K, V, qw = _snapkv_inputs(w, seed=6)
    batch = lib_batch(w, DEV)
    scores = torch.full(batch.score_shape(), float("nan"), dtype=torch.float32, device=DEV)
    R.quest_score(batch, qw, K, w.W, page, scores)
    torch.cuda.synchronize()
    ob = oracle_batch(w)
    qb, kb = I.bf16_bits(qw), I.bf16_bits(K)
    ref = O.quest_batch(ob, qb, kb, w.W, page)
    got_all = scores.cpu().numpy()
    for u, r in ref.items():
        got = ob.score_view(got_all, u).astype(np.float64)
        tol = 1e-5 * _quest_tol(ob, qb, kb, u, w.W, w.G) + 1e-4 * np.abs(r)
        assert np.all(np.abs(got - r) <= tol), f"{case} unit {u}"
        for p0 in range(0, got.size, page):          # one bound per page
            assert np.all(got[p0:p0 + page] == got[p0])
    # page top-k: the GLOBAL selector on the bounds keeps whole pages
    B = 0.10
    params = R.select_params(B, I.PAPER_ALPHA, 0.0, I.ROLE_KEY, policy=R.POLICY_GLOBAL)
    keep = torch.empty(batch.kept_shape(B), dtype=torch.int32, device=DEV)
    R.role_alloc_select(batch, scores, torch.as_tensor(roles_np, device=DEV), params, keep)
    torch.cuda.synchronize()
    keep_np, cu = keep.cpu().numpy(), ob.kept_offsets(B)
    for u, r in ref.items():
        l, s, h = ob.unit(u)
        row = keep_np[l, h, cu[s]:cu[s + 1]] if ob.varlen else keep_np.reshape(ob.n_units, -1)[u]
        check_index_sets(ob, u, row, r, roles_np, I.N_ROLES, I.PAPER_ALPHA, I.ROLE_KEY, 0.0, B,
                         policy=O.POLICY_GLOBAL)


# ------------------------------------------------------------------- decode

DECODE_CASES = {
    # name: (workload, budget, policy, ban_mask)
    "g4_b10": (_w("llama8b", L=2, b=2, Hq=8, Hkv=2, n=3001), 0.10, 0, 0),
    "d64": (_w("tiny", b=2), 0.30, 0, 0),
    "g7_varlen": (_w("ragged", L=1, b=3, Hq=14, Hkv=2, n=1500, seqlens=(1500, 31, 640)), 0.10, 0, 0),
    "varlen_empty_infeasible": (SNAPKV_CASES["varlen_short_empty"], 0.60, R.POLICY_GLOBAL,
                                ~(1 << I.ROLE_VALUE) & 0xF),
}


def _decode_ref(ob, w, qd_bits, kc, vc, valid_of):
    out = {}
    for u in range(ob.n_units):
        l, s, h = ob.unit(u)
        q = O.bf16_to_f64(qd_bits[l, s, h * w.G:(h + 1) * w.G])
        k, v, ok = kc(u), vc(u), valid_of(u)
        out[u] = O.decode_attention(q, O.bf16_to_f64(k), O.bf16_to_f64(v), ok, 1.0 / np.sqrt(w.d))
    return out


def _check_decode(ob, w, got, ref, vmax):
    g = got.cpu().numpy()
    for u, r in ref.items():
        l, s, h = ob.unit(u)
        o = g[l, s, h * w.G:(h + 1) * w.G].astype(np.float64)
        assert np.all(np.abs(o - r) <= 1e-3 * np.abs(r) + 1e-4 * vmax), f"unit {u}"


@pytest.mark.parametrize("case", list(DECODE_CASES))
def test_decode_attention_compacted(case):
    """Score -> select -> compact -> one decode step through the compacted
    cache, against the oracle on the compacted rows (-1 slots masked)."""
    w, B, policy, ban = DECODE_CASES[case]
    roles_np, K, V, qw = _snapkv_inputs(w, seed=7)
    batch = lib_batch(w, DEV)
    scores = torch.empty(batch.score_shape(), dtype=torch.float32, device=DEV)
    R.snapkv_score(batch, qw, K, w.W, w.pool_k, scores)
    keep = torch.empty(batch.kept_shape(B), dtype=torch.int32, device=DEV)
    R.role_alloc_select(batch, scores, torch.as_tensor(roles_np, device=DEV),
                        R.select_params(B, I.PAPER_ALPHA, 0.0, I.ROLE_KEY, policy=policy, ban_mask=ban),
                        keep)
    kc = torch.empty(R.compact_shape(batch, B), dtype=torch.bfloat16, device=DEV)
    vc = torch.empty_like(kc)
    R.kv_compact(batch, K, V, keep, B, kc, vc)
    qd = I.make_q_decode(w, 7, device=DEV)
    out = torch.full((w.L, w.b, w.Hq, w.d), float("nan"), dtype=torch.float32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    for _ in range(2):                               # the workspace holds no state
        R.decode_attention(batch, qd, kc, vc, keep, B, out, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ob = oracle_batch(w)
    kb, vb, kp = I.bf16_bits(kc), I.bf16_bits(vc), keep.cpu().numpy()
    cu = ob.kept_offsets(B)

    def rows(arr, u):
        l, s, h = ob.unit(u)
        return arr[l, h, cu[s]:cu[s + 1]] if ob.varlen else arr.reshape((ob.n_units, -1) + arr.shape[4:])[u]
    ref = _decode_ref(ob, w, I.bf16_bits(qd), lambda u: rows(kb, u), lambda u: rows(vb, u),
                      lambda u: rows(kp, u) >= 0)
    _check_decode(ob, w, out, ref, float(V.float().abs().max()))
    if case == "varlen_empty_infeasible":
        assert any((rows(kp, u) < 0).any() for u in range(ob.n_units))   # padding was exercised


@pytest.mark.parametrize("varlen", [False, True])
def test_decode_attention_full_cache(varlen):
    """Budget 1 and no index: attention over every cached token, in the
    uncompacted K/V layouts."""
    w = (SNAPKV_CASES["varlen_g7"] if varlen else _w("llama8b", L=1, b=2, Hq=8, Hkv=2, n=2000))
    roles_np, K, V, _ = _snapkv_inputs(w, seed=8)
    batch = lib_batch(w, DEV)
    qd = I.make_q_decode(w, 8, device=DEV)
    out = torch.empty((w.L, w.b, w.Hq, w.d), dtype=torch.float32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.decode_attention(batch, qd, K, V, None, 1.0, out, compacted=False, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ob = oracle_batch(w)
    kb, vb = I.bf16_bits(K), I.bf16_bits(V)
    ref = _decode_ref(ob, w, I.bf16_bits(qd), lambda u: ob.kv_rows(kb, u), lambda u: ob.kv_rows(vb, u),
                      lambda u: np.ones(ob.kv_rows(kb, u).shape[0], dtype=bool))
    _check_decode(ob, w, out, ref, float(V.float().abs().max()))


def test_decode_ignores_stale_stage_rows():
    """Rows past a unit's last cache row are never read into the result: a
    decode over a NaN-filled cache first leaves NaN bit patterns in the
    shared-memory stages, then a cache whose units end in a partial stage
    must still match the oracle."""
    w = _w("llama8b", L=2, b=2, Hq=8, Hkv=2, n=1999)
    roles_np, K, V, _ = _snapkv_inputs(w, seed=9)
    batch = lib_batch(w, DEV)
    qd = I.make_q_decode(w, 9, device=DEV)
    out = torch.empty((w.L, w.b, w.Hq, w.d), dtype=torch.float32, device=DEV)
    nan_k = torch.full_like(K, float("nan"))
    for _ in range(3):
        R.decode_attention(batch, qd, nan_k, nan_k, None, 1.0, out, compacted=False)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.decode_attention(batch, qd, K, V, None, 1.0, out, compacted=False, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert torch.isfinite(out).all()
    ob = oracle_batch(w)
    kb, vb = I.bf16_bits(K), I.bf16_bits(V)
    ref = _decode_ref(ob, w, I.bf16_bits(qd), lambda u: ob.kv_rows(kb, u), lambda u: ob.kv_rows(vb, u),
                      lambda u: np.ones(ob.kv_rows(kb, u).shape[0], dtype=bool))
    _check_decode(ob, w, out, ref, float(V.float().abs().max()))


# ------------------------------------------------------------------ selection

def _tied_scores(shape, seed):
    g = torch.Generator().manual_seed(seed)
    # coarse values create many exact ties, plateaus like a max-pool's
    return (torch.randint(0, 64, shape, generator=g).float() / 8.0).to(DEV)


VARLEN4 = _w("ragged", L=2, b=4, Hq=8, Hkv=2, n=3000, seqlens=(3000, 0, 5, 1200))
# longest row the selector holds in shared memory; longer rows stream their
# keys from the score row on every pass
SMEM_MAX_N = 40960
VARLEN_LONG = _w("ragged", L=1, b=4, Hq=4, Hkv=1, n=140000, seqlens=(140000, 0, 5, 50000))

SELECT_CASES = [
    # (name, workload, budget, alpha_key, policy, ban_mask, pool_k[, keep_last])
    ("combined_b05", _w("llama8b", L=2, b=2, Hq=8, Hkv=2, n=5000), 0.05, 0.0, 0, 0, 1),
    ("combined_b10_pool7", _w("llama8b", L=1, b=2, Hq=8, Hkv=2, n=5000), 0.10, 0.02, 0, 0, 7),
    ("combined_b50", _w("llama8b", L=1, b=1, Hq=8, Hkv=2, n=3001), 0.50, 0.0, 0, 0, 1),
    ("full_budget", _w("llama8b", L=1, b=1, Hq=4, Hkv=1, n=777), 1.0, 0.0, 0, 0, 3),
    ("global_no_key", _w("llama8b", L=1, b=2, Hq=8, Hkv=2, n=4000), 0.30, 0.0, 1, 1 << I.ROLE_KEY, 1),
    ("global_plain", _w("llama8b", L=1, b=1, Hq=8, Hkv=2, n=4000), 0.20, 0.0, 1, 0, 5),
    ("varlen", VARLEN4, 0.10, 0.0, 0, 0, 7),
    ("mid_n", _w("llama8b", L=1, b=1, Hq=8, Hkv=2, n=12001), 0.10, 0.02, 0, 0, 7),
    ("mid_n_global_pool15", _w("llama8b", L=1, b=1, Hq=4, Hkv=1, n=9999), 0.10, 0.0, 1, 0, 15),
    # the paper's other swept pool widths (Section 4: 3, 5, 7, 11, 15)
    ("combined_pool11", _w("llama8b", L=1, b=2, Hq=8, Hkv=2, n=5000), 0.10, 0.02, 0, 0, 11),
    ("varlen_global_pool11", VARLEN4, 0.20, 0.0, 1, 0, 11),
    ("max_n", _w("long", L=1, b=1, Hq=4, Hkv=1, n=SMEM_MAX_N), 0.10, 0.0, 0, 0, 7),
    # fair eviction (equal retention rate per role) and the recency floor
    ("fair_pool7", _w("llama8b", L=1, b=2, Hq=8, Hkv=2, n=5000), 0.10, 0.0, R.POLICY_FAIR, 0, 7),
    ("fair_no_key_varlen", VARLEN4, 0.20, 0.0, R.POLICY_FAIR, 1 << I.ROLE_KEY, 7),
    ("floor64_combined", _w("llama8b", L=1, b=2, Hq=8, Hkv=2, n=5000), 0.10, 0.02, 0, 0, 7, 64),
    ("floor32_global_varlen", VARLEN4, 0.10, 0.0, R.POLICY_GLOBAL, 0, 3, 32),
    ("floor_over_budget", _w("llama8b", L=1, b=1, Hq=8, Hkv=2, n=3001), 0.05, 0.0, 0, 0, 7, 1000),
    ("floor_fair_mid_n", _w("llama8b", L=1, b=1, Hq=8, Hkv=2, n=12001), 0.10, 0.0, R.POLICY_FAIR, 0, 7, 64),
    ("floor_max_n", _w("long", L=1, b=1, Hq=4, Hkv=1, n=SMEM_MAX_N), 0.10, 0.0, 0, 0, 7, 64),
    # role quotas with the slack of saturated buckets filled by score
    ("slack_b50", _w("llama8b", L=1, b=2, Hq=8, Hkv=2, n=5000), 0.50, 0.02, R.POLICY_SLACK, 0, 7),
    ("slack_b30_no_key_varlen", VARLEN4, 0.30, 0.0, R.POLICY_SLACK, 0, 7),
    ("slack_floor_mid_n", _w("llama8b", L=1, b=1, Hq=8, Hkv=2, n=12001), 0.20, 0.02, R.POLICY_SLACK, 0, 7, 64),
    ("slack_ban_max_n", _w("long", L=1, b=1, Hq=4, Hkv=1, n=SMEM_MAX_N), 0.30, 0.02, R.POLICY_SLACK,
     1 << I.ROLE_KEY, 1),
    # Algorithm 1's per-bucket ceilings taken literally (rows widened by
    # kept_extra = N_ROLES - 1 unless given), and widened rows under the exact split
    ("ceil_b10_pool7", _w("llama8b", L=1, b=2, Hq=8, Hkv=2, n=5000), 0.10, 0.02, R.POLICY_CEIL, 0, 7),
    ("ceil_varlen_floor32", VARLEN4, 0.05, 0.0, R.POLICY_CEIL, 0, 7, 32),
    ("ceil_ban_max_n", _w("long", L=1, b=1, Hq=4, Hkv=1, n=SMEM_MAX_N), 0.30, 0.02, R.POLICY_CEIL,
     1 << I.ROLE_KEY, 1),
    ("ceil_full_budget", _w("llama8b", L=1, b=1, Hq=4, Hkv=1, n=777), 1.0, 0.02, R.POLICY_CEIL, 0, 3),
    ("ceil_mid_n_extra9", _w("llama8b", L=1, b=1, Hq=8, Hkv=2, n=12001), 0.20, 0.02, R.POLICY_CEIL, 0, 7, 0, 9),
    ("quota_varlen_extra5", VARLEN4, 0.10, 0.02, 0, 0, 7, 0, 5),
    # rows past the shared-memory maximum (streaming mode), up to the ABI limit
    ("stream_65536", _w("long", L=1, b=1, Hq=4, Hkv=1, n=65536), 0.10, 0.02, 0, 0, 7),
    ("stream_131072_global_pool5", _w("long", L=1, b=1, Hq=4, Hkv=1, n=131072), 0.10, 0.0, 1, 0, 5),
    ("stream_131072_slack_floor", _w("long", L=1, b=1, Hq=4, Hkv=1, n=131072), 0.20, 0.02, R.POLICY_SLACK, 0,
     7, 64),
    ("stream_262144_ceil_pool3", _w("long", L=1, b=1, Hq=4, Hkv=1, n=R.SELECT_MAX_N), 0.05, 0.02,
     R.POLICY_CEIL, 0, 3),
    ("stream_varlen_fair", VARLEN_LONG, 0.10, 0.0, R.POLICY_FAIR, 1 << I.ROLE_KEY, 7),
    ("stream_varlen_quota_floor", VARLEN_LONG, 0.30, 0.02, 0, 0, 11, 32),
]


@pytest.mark.parametrize("case", SELECT_CASES, ids=[c[0] for c in SELECT_CASES])
def test_role_alloc_select_bit_exact(case):
    name, w, B, akey, policy, ban, pool_k = case[:7]
    keep_last = case[7] if len(case) > 7 else 0
    extra = case[8] if len(case) > 8 else (I.N_ROLES - 1 if policy == R.POLICY_CEIL else 0)
    roles_np = I.workload_roles(w, 2)
    batch = lib_batch(w, DEV, kept_extra=extra)
    scores = _tied_scores(batch.score_shape(), 5)
    roles = torch.as_tensor(roles_np, device=DEV)
    params = R.select_params(B, I.PAPER_ALPHA, alpha_key=akey, key_role=I.ROLE_KEY, policy=policy,
                             ban_mask=ban, keep_last=keep_last)
    keep = torch.full(batch.kept_shape(B), -7, dtype=torch.int32, device=DEV)
    mask = torch.full(batch.score_shape(), 9, dtype=torch.uint8, device=DEV)
    per_role = torch.full((batch.n_units, I.N_ROLES), -1, dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.role_alloc_select(batch, scores, roles, params, keep, pool_k=pool_k, keep_mask=mask,
                        kept_per_role=per_role, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ob = oracle_batch(w, kept_extra=extra)
    sc = scores.cpu().numpy()
    unit_scores = {}
    for u in range(ob.n_units):
        s = ob.score_view(sc, u).astype(np.float64)
        unit_scores[u] = O.maxpool1d(s, pool_k) if s.size else s
    ref = O.select_batch(ob, unit_scores, roles_np, I.N_ROLES, I.PAPER_ALPHA, I.ROLE_KEY, akey, B,
                         policy, ban, keep_last=keep_last)
    cu_kept = ob.kept_offsets(B)
    keep_np, mask_np, pr = keep.cpu().numpy(), mask.cpu().numpy(), per_role.cpu().numpy()
    for u, (idx, per) in ref.items():
        l, s, h = ob.unit(u)
        if ob.varlen:
            row = keep_np[l, h, cu_kept[s]:cu_kept[s + 1]]
        else:
            row = keep_np.reshape(ob.n_units, -1)[u]
        assert np.array_equal(row, idx), f"{name} unit {u}"
        assert list(pr[u]) == per, f"{name} unit {u} per-role counts"
        m = ob.score_view(mask_np, u)
        expect = np.zeros(m.shape, dtype=np.uint8)
        expect[idx[idx >= 0]] = 1
        assert np.array_equal(m, expect), f"{name} unit {u} mask"
        if akey == 0.0 and policy == 0 and keep_last == 0:
            assert per[I.ROLE_KEY] == 0


NARROW_CASES = [
    # (name, n, policy, pool_k, spread[, budget]): page-constant scores in [2, 2 + spread)
    ("narrow_quota", 20000, 0, 1, 0.2),
    ("narrow_global_stream", 70000, 1, 3, 0.2),
    ("narrow_global_pool7", 20000, 1, 7, 0.2),
    ("narrow_fair_short", 9000, 2, 1, 0.2),
    ("constant_global", 20000, 1, 1, 0.0),
    ("constant_quota_pool5", 12000, 0, 5, 0.0),
    # SLACK fill: its first digit holds a few thousand page-tied keys (listed,
    # then ranked), or every key (the list overflows: full-pass rounds)
    ("narrow_slack_b50", 20000, 3, 1, 2.0, 0.5),
    ("constant_slack_pool3_b50", 16000, 3, 3, 0.0, 0.5),
]


@pytest.mark.parametrize("case", NARROW_CASES, ids=[c[0] for c in NARROW_CASES])
def test_select_narrow_page_constant_scores(case):
    """Scores constant over pages of 16 and packed into a narrow range (as
    Quest page bounds are): most keys share the first digit, so the selector
    takes extra digit rounds before listing candidates; a constant row leaves
    only ties.  Bit-exact against the oracle on the same scores."""
    name, n, policy, pool_k, spread = case[:5]
    B = case[5] if len(case) > 5 else 0.10
    w = _w("llama8b", L=1, b=2, Hq=8, Hkv=2, n=n)
    roles_np = I.workload_roles(w, 3)
    batch = lib_batch(w, DEV)
    g = torch.Generator().manual_seed(17)
    npages = (n + 15) // 16
    pages = 2.0 + spread * torch.rand((batch.n_units, npages), generator=g)
    sc = pages.repeat_interleave(16, dim=1)[:, :n].reshape(batch.score_shape()).contiguous()
    scores = sc.to(DEV)
    params = R.select_params(B, I.PAPER_ALPHA, alpha_key=0.0, key_role=I.ROLE_KEY, policy=policy)
    keep = torch.full(batch.kept_shape(B), -7, dtype=torch.int32, device=DEV)
    per_role = torch.full((batch.n_units, I.N_ROLES), -1, dtype=torch.int32, device=DEV)
    R.role_alloc_select(batch, scores, torch.as_tensor(roles_np, device=DEV), params, keep,
                        pool_k=pool_k, kept_per_role=per_role)
    torch.cuda.synchronize()
    ob = oracle_batch(w)
    scn = sc.numpy()
    unit_scores = {u: O.maxpool1d(ob.score_view(scn, u).astype(np.float64), pool_k)
                   for u in range(ob.n_units)}
    ref = O.select_batch(ob, unit_scores, roles_np, I.N_ROLES, I.PAPER_ALPHA, I.ROLE_KEY, 0.0, B,
                         policy)
    got, pr = keep.cpu().numpy().reshape(ob.n_units, -1), per_role.cpu().numpy()
    for u, (idx, per) in ref.items():
        assert np.array_equal(got[u], idx), f"{name} unit {u}"
        assert list(pr[u]) == per, f"{name} unit {u} per-role counts"


@pytest.mark.parametrize("akey", [0.0, 0.02])
def test_select_six_role_taxonomy(akey):
    """The paper's six labels (KEY, VALUE, DELIM, HEADER, PROSE, WS) with its
    policy; a few tokens carry labels outside the six (no bucket)."""
    w = _w("llama8b", L=1, b=2, Hq=8, Hkv=2, n=6001)
    g = np.random.default_rng(8)
    roles_np = g.choice(8, size=(w.b, w.n), p=[0.25, 0.2, 0.3, 0.05, 0.1, 0.08, 0.01, 0.01]).astype(np.uint8)
    batch = lib_batch(w, DEV)
    scores = _tied_scores(batch.score_shape(), 13)
    alpha = I.paper_alpha6(akey)
    B = 0.10
    params = R.select_params(B, alpha, alpha_key=akey, key_role=0)
    keep = torch.empty(batch.kept_shape(B), dtype=torch.int32, device=DEV)
    per_role = torch.empty((batch.n_units, 6), dtype=torch.int32, device=DEV)
    R.role_alloc_select(batch, scores, torch.as_tensor(roles_np, device=DEV), params, keep, pool_k=7,
                        kept_per_role=per_role)
    torch.cuda.synchronize()
    ob = oracle_batch(w)
    sc = scores.cpu().numpy()
    unit_scores = {u: O.maxpool1d(ob.score_view(sc, u).astype(np.float64), 7) for u in range(ob.n_units)}
    ref = O.select_batch(ob, unit_scores, roles_np, 6, alpha, 0, akey, B)
    got, pr = keep.cpu().numpy().reshape(ob.n_units, -1), per_role.cpu().numpy()
    for u, (idx, per) in ref.items():
        assert np.array_equal(got[u], idx), f"unit {u}"
        assert list(pr[u]) == per
        if akey == 0.0:
            assert per[0] == 0 and per[3] == 0


@pytest.mark.parametrize("pool_k,n", [(1, 3001), (7, 3001), (5, 50001)])
def test_select_nan_scores_flagged_and_lowest(pool_k, n):
    """A NaN score sets STATUS_NONFINITE; every pooled window holding a NaN
    ranks below every other token (kept last, ties in index order); also in
    the streaming mode (n above the shared-memory maximum)."""
    w = _w("llama8b", L=1, b=2, Hq=4, Hkv=1, n=n)
    roles_np = I.workload_roles(w, 4)
    batch = lib_batch(w, DEV)
    g = torch.Generator().manual_seed(11)
    sc = torch.rand(batch.score_shape(), generator=g)
    flat = sc.view(-1)
    flat[torch.randint(0, flat.numel(), (40,), generator=g)] = float("nan")
    B = 0.60
    keep = torch.empty(batch.kept_shape(B), dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.role_alloc_select(batch, sc.to(DEV), torch.as_tensor(roles_np, device=DEV),
                        R.select_params(B, I.PAPER_ALPHA, 0.0, I.ROLE_KEY), keep, pool_k=pool_k,
                        status=status)
    torch.cuda.synchronize()
    assert int(status.item()) & R.STATUS_NONFINITE
    ob = oracle_batch(w)
    sc_np = sc.numpy()
    unit_scores = {}
    for u in range(ob.n_units):
        x = ob.score_view(sc_np, u).astype(np.float64)
        hw = pool_k // 2
        nan_win = np.array([np.isnan(x[max(0, t - hw):t + hw + 1]).any() for t in range(x.size)])
        pooled = O.maxpool1d(np.where(np.isnan(x), -np.inf, x), pool_k)
        unit_scores[u] = np.where(nan_win, -np.inf, pooled)
    ref = O.select_batch(ob, unit_scores, roles_np, I.N_ROLES, I.PAPER_ALPHA, I.ROLE_KEY, 0.0, B)
    got = keep.cpu().numpy().reshape(ob.n_units, -1)
    for u, (idx, _) in ref.items():
        assert np.array_equal(got[u], idx), f"unit {u}"


def test_select_infeasible_budget_pads():
    """More budget than eligible tokens: every eligible token is kept and the
    tail of the row is -1."""
    w = _w("llama8b", L=1, b=1, Hq=4, Hkv=1, n=600)
    roles_np = np.full((1, 600), I.ROLE_KEY, dtype=np.uint8)
    roles_np[0, ::10] = I.ROLE_VALUE
    batch = lib_batch(w, DEV)
    scores = _tied_scores(batch.score_shape(), 9)
    keep = torch.empty(batch.kept_shape(0.5), dtype=torch.int32, device=DEV)
    R.role_alloc_select(batch, scores, torch.as_tensor(roles_np, device=DEV),
                        R.select_params(0.5, I.PAPER_ALPHA, 0.0, I.ROLE_KEY), keep)
    torch.cuda.synchronize()
    row = keep.cpu().numpy().reshape(-1)
    assert row.size == 300
    assert np.array_equal(row[:60], np.arange(0, 600, 10))
    assert np.all(row[60:] == -1)


# ----------------------------------------------------------------- compaction

@pytest.mark.parametrize("varlen", [False, True])
def test_kv_compact_bit_exact(varlen):
    if varlen:
        w = _w("ragged", L=2, b=3, Hq=8, Hkv=2, n=900, seqlens=(900, 0, 333))
    else:
        w = _w("llama8b", L=2, b=2, Hq=8, Hkv=2, n=1000)
    B = 0.2
    roles = I.workload_roles(w, 4)
    K, V = I.make_kv(w, roles, 4, device=DEV)
    batch = lib_batch(w, DEV)
    rng = np.random.default_rng(11)
    keep_np = np.full(batch.kept_shape(B), -1, dtype=np.int32)
    ob = oracle_batch(w)
    cu_kept = ob.kept_offsets(B)
    for u in range(ob.n_units):
        l, s, h = ob.unit(u)
        n = ob.seqlens[s]
        kcount = O.kept_count(n, B) if n else 0
        take = max(0, kcount - 3)
        idx = np.sort(rng.choice(n, size=take, replace=False)) if take else np.zeros(0, int)
        row = np.full(kcount, -1, dtype=np.int32)
        row[:take] = idx
        if varlen:
            keep_np[l, h, cu_kept[s]:cu_kept[s + 1]] = row
        else:
            keep_np.reshape(ob.n_units, -1)[u] = row
    keep = torch.as_tensor(keep_np, device=DEV)
    k_out = torch.full(R.compact_shape(batch, B), 3.0, dtype=torch.bfloat16, device=DEV)
    v_out = torch.full_like(k_out, 3.0)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    R.kv_compact(batch, K, V, keep, B, k_out, v_out, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    kb, vb = I.bf16_bits(K), I.bf16_bits(V)
    ko, vo = I.bf16_bits(k_out), I.bf16_bits(v_out)
    for u in range(ob.n_units):
        l, s, h = ob.unit(u)
        if varlen:
            sl = slice(cu_kept[s], cu_kept[s + 1])
            row, kr, vr = keep_np[l, h, sl], ko[l, h, sl], vo[l, h, sl]
        else:
            row = keep_np.reshape(ob.n_units, -1)[u]
            kr = ko.reshape(ob.n_units, -1, w.d)[u]
            vr = vo.reshape(ob.n_units, -1, w.d)[u]
        assert np.array_equal(kr, O.compact_unit(ob.kv_rows(kb, u), row))
        assert np.array_equal(vr, O.compact_unit(ob.kv_rows(vb, u), row))
        ok = row >= 0
        ref_t = torch.index_select(torch.as_tensor(ob.kv_rows(kb, u).astype(np.int32)), 0,
                                   torch.as_tensor(row[ok].astype(np.int64)))
        assert np.array_equal(kr[ok].astype(np.int32), ref_t.numpy())


def test_kv_compact_reads_pinned_host_values():
    """V left in pinned host memory: the compaction gathers the kept rows
    across the host link and writes exactly what it writes from device V."""
    w = _w("ragged", L=2, b=3, Hq=8, Hkv=2, n=900, seqlens=(900, 0, 333))
    B = 0.2
    roles = I.workload_roles(w, 5)
    K, V = I.make_kv(w, roles, 5, device=DEV)
    batch = lib_batch(w, DEV)
    ob = oracle_batch(w)
    rng = np.random.default_rng(12)
    keep_np = np.full(batch.kept_shape(B), -1, dtype=np.int32)
    cu_kept = ob.kept_offsets(B)
    for u in range(ob.n_units):
        l, s, h = ob.unit(u)
        n, k = ob.seqlens[s], int(cu_kept[s + 1] - cu_kept[s])
        if k:
            keep_np[l, h, cu_kept[s]:cu_kept[s] + k - 1] = np.sort(rng.choice(n, size=k - 1, replace=False))
    keep = torch.as_tensor(keep_np, device=DEV)
    h_v = torch.empty(V.shape, dtype=V.dtype, pin_memory=True)
    h_v.copy_(V)
    outs = []
    for vv in (V, h_v):
        k_out = torch.full(R.compact_shape(batch, B), 3.0, dtype=torch.bfloat16, device=DEV)
        v_out = torch.full_like(k_out, 3.0)
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        R.kv_compact(batch, K, vv, keep, B, k_out, v_out, status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        outs.append((k_out, v_out))
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])
    vb, vo = I.bf16_bits(V), I.bf16_bits(outs[1][1])
    for u in range(ob.n_units):
        l, s, h = ob.unit(u)
        sl = slice(cu_kept[s], cu_kept[s + 1])
        assert np.array_equal(vo[l, h, sl], O.compact_unit(ob.kv_rows(vb, u), keep_np[l, h, sl]))


# ------------------------------------------------------------- whole pipeline

@pytest.mark.parametrize("name", ["tiny", "ragged_small", "ragged_small_ceil"])
def test_rolekv_compress_pipeline(name):
    if name == "tiny":
        w = I.WORKLOADS["tiny"]
    else:
        w = _w("ragged", L=2, b=4, Hq=14, Hkv=2, n=3000, seqlens=(3000, 1024, 77, 2222))
    B = w.budgets[0]
    policy = R.POLICY_CEIL if name.endswith("ceil") else R.POLICY_ROLE_QUOTA
    extra = I.N_ROLES - 1 if policy == R.POLICY_CEIL else 0
    roles_np, K, V, qw = _snapkv_inputs(w, seed=6)
    batch = lib_batch(w, DEV, kept_extra=extra)
    params = R.select_params(B, I.PAPER_ALPHA, 0.0, I.ROLE_KEY, policy=policy)
    keep = torch.empty(batch.kept_shape(B), dtype=torch.int32, device=DEV)
    k_out = torch.empty(R.compact_shape(batch, B), dtype=torch.bfloat16, device=DEV)
    v_out = torch.empty_like(k_out)
    ws = R.workspace(R.OP_COMPRESS, batch, w.W)
    roles = torch.as_tensor(roles_np, device=DEV)
    R.rolekv_compress(batch, qw, K, V, w.W, w.pool_k, roles, params, keep, k_out, v_out, ws)
    # the separate calls give the same kept set
    scores = torch.empty(batch.score_shape(), dtype=torch.float32, device=DEV)
    R.snapkv_score(batch, qw, K, w.W, w.pool_k, scores)
    keep2 = torch.empty_like(keep)
    R.role_alloc_select(batch, scores, roles, params, keep2)
    torch.cuda.synchronize()
    assert torch.equal(keep, keep2)
    ob = oracle_batch(w, kept_extra=extra)
    ref = O.snapkv_batch(ob, I.bf16_bits(qw), I.bf16_bits(K), w.W, w.pool_k)
    cu_kept = ob.kept_offsets(B)
    keep_np = keep.cpu().numpy()
    ko = I.bf16_bits(k_out)
    kb = I.bf16_bits(K)
    for u, (_, pooled) in ref.items():
        l, s, h = ob.unit(u)
        if ob.varlen:
            row = keep_np[l, h, cu_kept[s]:cu_kept[s + 1]]
            kr = ko[l, h, cu_kept[s]:cu_kept[s + 1]]
        else:
            row = keep_np.reshape(ob.n_units, -1)[u]
            kr = ko.reshape(ob.n_units, -1, w.d)[u]
        check_index_sets(ob, u, row, pooled, roles_np, I.N_ROLES, I.PAPER_ALPHA, I.ROLE_KEY, 0.0, B,
                         policy)
        assert np.array_equal(kr, O.compact_unit(ob.kv_rows(kb, u), row))


def test_bounded_wait_reports_timeout():
    """A device wait that nothing satisfies gives up after its limit, records
    STATUS_TIMEOUT, and leaves the context usable for the next launch."""
    import time
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    R.selftest_wait(20_000_000, status)          # 20 ms
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    assert int(status.item()) & R.STATUS_TIMEOUT
    assert 0.015 <= dt < 5.0
    x = torch.arange(8, device=DEV).sum()        # the context still works
    assert int(x.item()) == 28


@pytest.mark.parametrize("case", ["two_row_tiles_w64_multichunk", "varlen_short_empty"])
def test_fused_score_meeting_point_timeout(case):
    """The persistent score kernel's own abort path: armed by the self-test,
    its per-unit meeting point waits for an arrival that never comes, gives up
    after 30 ms, reports STATUS_TIMEOUT and returns (its copies drained, its
    tensor memory freed).  The next call on the same device and stream runs
    normally and matches the oracle."""
    import time
    w = SNAPKV_CASES[case]
    roles, K, V, qw = _snapkv_inputs(w, seed=12)
    batch = lib_batch(w, DEV)
    scores = torch.full(batch.score_shape(), -1.0, dtype=torch.float32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    R.selftest_score_timeout(30_000_000)
    R.snapkv_score(batch, qw, K, w.W, 1, scores, status=status)
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    assert int(status.item()) & R.STATUS_TIMEOUT
    assert 0.025 <= dt < 10.0
    # the arming is used up: the next call is a normal one
    status.zero_()
    R.snapkv_score(batch, qw, K, w.W, 1, scores, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ob = oracle_batch(w)
    ref = O.snapkv_batch(ob, I.bf16_bits(qw), I.bf16_bits(K), w.W, 1)
    got = scores.cpu().numpy()
    for u, (rpre, _) in ref.items():
        assert_scores_close(ob.score_view(got, u), rpre, f"{case} unit {u} after the timeout")


@pytest.mark.parametrize("varlen", [False, True])
def test_layer_slices_match_whole_batch(varlen):
    """The calls on layer slices of the tensors (views with a storage offset,
    a batch of fewer layers) give exactly the whole batch's scores, kept
    indices and compressed rows, as a prefill handing over its cache layer by
    layer would use them."""
    w = (_w("ragged", L=4, b=3, Hq=8, Hkv=2, n=2000, seqlens=(2000, 700, 0)) if varlen
         else _w("llama8b", L=4, b=2, Hq=8, Hkv=2, n=2500))
    roles_np, K, V, qw = _snapkv_inputs(w, seed=11)
    roles = torch.as_tensor(roles_np, device=DEV)
    B = 0.1
    params = R.select_params(B, I.PAPER_ALPHA, 0.02, I.ROLE_KEY)
    full = lib_batch(w, DEV)

    def run(batch, q, k, v):
        sc = torch.empty(batch.score_shape(), dtype=torch.float32, device=DEV)
        R.snapkv_score(batch, q, k, w.W, 1, sc)
        kp = torch.empty(batch.kept_shape(B), dtype=torch.int32, device=DEV)
        R.role_alloc_select(batch, sc, roles, params, kp, pool_k=w.pool_k)
        ko = torch.empty(R.compact_shape(batch, B), dtype=torch.bfloat16, device=DEV)
        vo = torch.empty_like(ko)
        R.kv_compact(batch, k, v, kp, B, ko, vo)
        return sc, kp, ko, vo

    whole = run(full, qw, K, V)
    half = _w(w.name, **{f: getattr(w, f) for f in ("b", "Hq", "Hkv", "d", "n", "W", "pool_k", "seqlens")},
              L=2)
    sb = lib_batch(half, DEV)
    parts = [run(sb, qw[l0:l0 + 2], K[l0:l0 + 2], V[l0:l0 + 2]) for l0 in (0, 2)]
    torch.cuda.synchronize()
    for x, (a, b) in enumerate(zip(whole, zip(*parts))):
        assert torch.equal(torch.cat(b, dim=0), a), f"output {x}"
