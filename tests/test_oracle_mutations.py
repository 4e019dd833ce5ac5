"""Plant plausible mistakes in a private copy of the oracle (on the CPU) and
check that at least one pin catches each of them."""
import importlib.util
import math
import os

import numpy as np
import pytest

from tests import oracle_pins as P

ORACLE_FILE = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                           "oracle", "rolekv_oracle.py")


def _fresh_oracle(tag):
    spec = importlib.util.spec_from_file_location(f"_mutant_oracle_{tag}", ORACLE_FILE)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _probs_factory(mask_rule="causal", scale_pow=1, norm_axis=1):
    def attention_probs(q_rows, k, positions, scale):
        q_rows = np.asarray(q_rows, dtype=np.float64)
        k = np.asarray(k, dtype=np.float64)
        n = k.shape[0]
        logits = (scale ** scale_pow) * (q_rows @ k.T)
        t = np.arange(n)[None, :]
        p = np.asarray(positions)[:, None]
        if mask_rule == "causal":
            vis = t <= p
        elif mask_rule == "strict":
            vis = t < p
            vis[:, 0] = True
        else:
            vis = np.ones_like(t <= p)
        logits = np.where(vis, logits, -np.inf)
        m = logits.max(axis=1, keepdims=True)
        e = np.where(vis, np.exp(logits - m), 0.0)
        return e / e.sum(axis=norm_axis, keepdims=True)
    return attention_probs


def _m_no_causal(O):
    O.attention_probs = _probs_factory(mask_rule="none")


def _m_strict_causal(O):
    O.attention_probs = _probs_factory(mask_rule="strict")


def _m_scale_squared(O):
    O.attention_probs = _probs_factory(scale_pow=2)


def _m_column_normalised(O):
    O.attention_probs = _probs_factory(norm_axis=0)


def _m_first_window(O):
    O.window_positions = lambda n, W: np.arange(0, min(W, n))
    orig = O.snapkv_prepool

    def snapkv_prepool(q_win, k, W, scale):
        n = k.shape[0]
        w_eff = min(W, n)
        pos = np.arange(0, w_eff)
        s = np.zeros(n)
        for g in range(q_win.shape[0]):
            s += O.attention_probs(q_win[g, :w_eff, :], k, pos, scale).sum(axis=0)
        return s
    O.snapkv_prepool = snapkv_prepool
    del orig


def _m_mean_over_heads(O):
    orig = O.snapkv_prepool
    O.snapkv_prepool = lambda q_win, k, W, scale: orig(q_win, k, W, scale) / q_win.shape[0]


def _m_h2o_drops_heads(O):
    orig = O.h2o_score
    O.h2o_score = lambda q, k, scale, row_block=2048: orig(q[:1], k, scale, row_block)


def _m_pool_too_wide(O):
    def maxpool1d(s, kernel):
        s = np.asarray(s, dtype=np.float64)
        n, h = s.shape[0], kernel // 2 + 1
        return np.array([s[max(0, t - h): min(n, t + h + 1)].max() for t in range(n)])
    O.maxpool1d = maxpool1d


def _m_pool_one_sided(O):
    def maxpool1d(s, kernel):
        s = np.asarray(s, dtype=np.float64)
        n = s.shape[0]
        return np.array([s[t: min(n, t + kernel)].max() for t in range(n)])
    O.maxpool1d = maxpool1d


def _m_round_not_ceil(O):
    def kept_count(n, budget):
        b = O.to_fixed(budget)
        return (b * n + O.FIXED_ONE // 2) // O.FIXED_ONE
    O.kept_count = kept_count


def _m_no_redistribution(O):
    def role_quotas(counts, alpha, budget, n, policy=0, ban_mask=0, k_full=None):
        R = len(counts)
        a = [O.to_fixed(x) for x in alpha]
        E = [r for r in range(R) if a[r] > 0 and counts[r] > 0]
        kf = O.kept_count(n, budget) if k_full is None else k_full
        K = min(kf, sum(counts[r] for r in E))
        A = sum(a[r] for r in E) or 1
        q = [0] * R
        for r in E:
            q[r] = min(counts[r], math.ceil(a[r] * K / A))
        return q
    O.role_quotas = role_quotas


def _m_renormalise_all_buckets(O):
    orig = O.role_quotas

    def role_quotas(counts, alpha, budget, n, policy=0, ban_mask=0, k_full=None):
        # shares computed over every bucket with alpha > 0, present or not
        R = len(counts)
        a = [O.to_fixed(x) for x in alpha]
        kf = O.kept_count(n, budget) if k_full is None else k_full
        K = min(kf, sum(c for c, x in zip(counts, a) if x > 0))
        A = sum(a) or 1
        q = [min(counts[r], (a[r] * K) // A) for r in range(R)]
        return q
    O.role_quotas = role_quotas
    del orig


def _m_remainder_ties_high(O):
    src = open(ORACLE_FILE).read().replace("key=lambda r: (-rem[r], r)", "key=lambda r: (-rem[r], -r)")
    ns = {}
    exec(compile(src, ORACLE_FILE, "exec"), ns)
    O.role_quotas = ns["role_quotas"]


def _m_ties_to_high_index(O):
    def select_unit(scores, buckets, quotas):
        scores = np.asarray(scores, dtype=np.float64)
        kept = []
        for r, qr in enumerate(quotas):
            if qr <= 0:
                continue
            idx = np.nonzero(buckets == r)[0]
            order = np.lexsort((-idx, -scores[idx]))
            kept.append(idx[order[:qr]])
        return np.sort(np.concatenate(kept)) if kept else np.zeros(0, dtype=np.int64)
    O.select_unit = select_unit


def _m_interleaved_gqa(O):
    def snapkv_batch(batch, q_win_bits, k_bits, W, pool_k, scale=None, units=None):
        scale = 1.0 / math.sqrt(batch.d) if scale is None or scale <= 0 else scale
        out = {}
        for u in (range(batch.n_units) if units is None else units):
            l, s, h = batch.unit(u)
            k = O.bf16_to_f64(batch.kv_rows(k_bits, u))
            heads = [h + batch.Hkv * g for g in range(batch.G)]
            qw = O.bf16_to_f64(q_win_bits[l, s, heads, :, :])
            pre = O.snapkv_prepool(qw, k, W, scale)
            out[u] = (pre, O.maxpool1d(pre, pool_k))
        return out
    O.snapkv_batch = snapkv_batch


def _from_source(O, old, new, names):
    src = open(ORACLE_FILE).read()
    assert old in src, old
    ns = {}
    exec(compile(src.replace(old, new), ORACLE_FILE, "exec"), ns)
    for nm in names:
        setattr(O, nm, ns[nm])


def _m_fair_uses_alpha(O):
    _from_source(O, "a = [0 if (ban_mask >> r) & 1 else counts[r] for r in range(R)]",
                 "a = [0 if (ban_mask >> r) & 1 else to_fixed(alpha[r]) for r in range(R)]",
                 ["role_quotas"])


def _m_floor_outside_budget(O):
    _from_source(O, "k_full=budget_n - forced)", "k_full=budget_n)", ["select_batch"])


def _m_floor_counts_whole_row(O):
    _from_source(O, "counts = [int((r[:nf] == x).sum())", "counts = [int((r == x).sum())",
                 ["select_batch"])


def _m_quest_max_only(O):
    _from_source(O, "np.maximum(qbar * lo, qbar * hi).sum()", "(qbar * hi).sum()", ["quest_score"])


def _m_quest_window_start(O):
    _from_source(O, "q = np.asarray(q_win, dtype=np.float64)[:, :w_eff, :]",
                 "q = np.asarray(q_win, dtype=np.float64)", ["quest_score"])


def _m_quest_exact_page_max(O):
    # the exact best dot product of the page: also an upper bound, exact for
    # one-token pages and for equal keys, but not Quest's per-dimension bound
    _from_source(O, "np.maximum(qbar * lo, qbar * hi).sum()", "(blk @ qbar).max()", ["quest_score"])


def _m_decode_scale_squared(O):
    _from_source(O, "logits = scale * (q @ kk.T)", "logits = scale * scale * (q @ kk.T)",
                 ["decode_attention"])


def _m_decode_no_scale(O):
    _from_source(O, "logits = scale * (q @ kk.T)", "logits = (q @ kk.T)", ["decode_attention"])


def _m_decode_keeps_padding(O):
    _from_source(O, "kk, vv = k[valid], v[valid]", "kk, vv = k, v", ["decode_attention"])


def _m_decode_unnormalised(O):
    _from_source(O, "return (e / e.sum(axis=1, keepdims=True)) @ vv", "return e @ vv", ["decode_attention"])


def _m_slack_from_all_roles(O):
    _from_source(O, "pool = np.nonzero(np.isin(r[:nf], E))[0]", "pool = np.arange(nf)", ["select_batch"])


def _m_slack_waterfills(O):
    _from_source(O, "while S and policy != POLICY_SLACK:", "while S:", ["role_quotas"])


def _m_slack_not_filled(O):
    _from_source(O, "if slack > 0:", "if slack > 10**9:", ["select_batch"])


def _m_ceil_floors(O):
    _from_source(O, "q[r] = -((-a[r] * k_left) // A)", "q[r] = (a[r] * k_left) // A", ["role_quotas"])


def _m_ceil_no_waterfill(O):
    _from_source(O, "while S and policy != POLICY_SLACK:", "while S and policy not in (POLICY_SLACK, POLICY_CEIL):",
                 ["role_quotas"])


def _m_ceil_unnormalised(O):
    _from_source(O, "q[r] = -((-a[r] * k_left) // A)", "q[r] = -((-a[r] * k_left) // FIXED_ONE)", ["role_quotas"])


def _m_ceil_rows_not_widened(O):
    _from_source(O, "width = batch.kept_rows(n, budget)", "width = budget_n", ["select_batch"])


def _m_compact_off_by_one(O):
    orig = O.compact_unit
    O.compact_unit = lambda rows, idx: orig(rows, np.where(np.asarray(idx) >= 0, np.minimum(np.asarray(idx) + 1, rows.shape[0] - 1), -1))


MUTATIONS = [
    _m_no_causal, _m_strict_causal, _m_scale_squared, _m_column_normalised, _m_first_window,
    _m_mean_over_heads, _m_h2o_drops_heads, _m_pool_too_wide, _m_pool_one_sided,
    _m_round_not_ceil, _m_no_redistribution, _m_renormalise_all_buckets, _m_remainder_ties_high,
    _m_ties_to_high_index, _m_interleaved_gqa, _m_compact_off_by_one, _m_fair_uses_alpha,
    _m_floor_outside_budget, _m_floor_counts_whole_row, _m_quest_max_only, _m_quest_window_start,
    _m_quest_exact_page_max, _m_decode_scale_squared, _m_decode_no_scale,
    _m_decode_keeps_padding, _m_decode_unnormalised, _m_slack_from_all_roles, _m_slack_waterfills,
    _m_slack_not_filled, _m_ceil_floors, _m_ceil_no_waterfill, _m_ceil_unnormalised,
    _m_ceil_rows_not_widened,
]


@pytest.mark.parametrize("mutate", MUTATIONS, ids=lambda f: f.__name__[3:])
def test_planted_mistake_is_caught(mutate):
    O = _fresh_oracle(mutate.__name__)
    mutate(O)
    caught = []
    for pin in P.ALL_PINS:
        try:
            pin(O, np.random.default_rng(20260713))
        except Exception as exc:  # noqa: BLE001 - any failure counts as caught
            caught.append((pin.__name__, type(exc).__name__))
    assert caught, f"no pin caught mutation {mutate.__name__}"
