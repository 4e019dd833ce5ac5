"""Pins of the fp64 oracle against facts fixed by the paper and by mathematics.

Each ``pin_*`` takes the oracle module (so the same checks can be run on a
copy of it with a planted mistake) and raises AssertionError on a violation.
None of them re-types the oracle's formula: they use closed forms, invariants,
hand-worked values (``tests/golden``), independent formulations and library
routines for special cases.
"""

from __future__ import annotations

import itertools
import json
import math
import os
from fractions import Fraction

import numpy as np
from scipy.ndimage import maximum_filter1d

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _bf16_bits(x):
    """float -> bf16 bits, for values that are exactly representable."""
    f = np.asarray(x, dtype=np.float32)
    bits = f.view(np.uint32)
    assert np.all((bits & 0xFFFF) == 0), "value not exact in bf16"
    return (bits >> 16).astype(np.uint16)


def _harmonic(m):
    return sum(Fraction(1, j) for j in range(1, m + 1))


# ---------------------------------------------------------------- softmax ---

def pin_rows_sum_to_one(O, rng):
    """Every causal softmax row sums to 1 and puts no mass after its position."""
    n, d = 57, 16
    q = rng.standard_normal((9, d)) * 2
    k = rng.standard_normal((n, d)) * 2
    pos = np.array([0, 3, 10, 20, 33, 40, 50, 55, 56])
    P = O.attention_probs(q, k, pos, 1 / math.sqrt(d))
    assert np.allclose(P.sum(axis=1), 1.0, rtol=0, atol=1e-12)
    for r, p in enumerate(pos):
        assert np.all(P[r, p + 1:] == 0)
        assert np.all(P[r, :p + 1] > 0)


def pin_snapkv_total(O, rng):
    """SnapKV pre-pool mass of a unit totals W_eff * G (every window row is a
    probability distribution), for W < n and W > n."""
    d, G = 16, 3
    for n, W in ((40, 8), (5, 8), (64, 64)):
        qw = rng.standard_normal((G, W, d))
        k = rng.standard_normal((n, d))
        s = O.snapkv_prepool(qw, k, W, 1 / math.sqrt(d))
        assert s.shape == (n,)
        assert abs(s.sum() - min(W, n) * G) < 1e-10


def pin_h2o_total(O, rng):
    """H2O mass of a unit totals n * G (one distribution per causal query)."""
    d, G, n = 16, 2, 37
    q = rng.standard_normal((G, n, d))
    k = rng.standard_normal((n, d))
    s = O.h2o_score(q, k, 1 / math.sqrt(d))
    assert abs(s.sum() - n * G) < 1e-10


def pin_uniform_closed_forms(O, rng):
    """Identical keys give uniform attention over each causal prefix, so
    SnapKV s(t) = G * sum over window positions p >= t of 1/(p+1) and
    H2O s(t) = G * (H_n - H_t), H the harmonic numbers."""
    d, G, n, W = 8, 2, 23, 6
    k = np.tile(rng.standard_normal(d), (n, 1))
    qw = rng.standard_normal((G, W, d))
    s = O.snapkv_prepool(qw, k, W, 1 / math.sqrt(d))
    window = range(n - W, n)
    for t in range(n):
        exact = G * sum(Fraction(1, p + 1) for p in window if p >= t)
        assert abs(s[t] - float(exact)) < 1e-12, (t, s[t], float(exact))
    q = rng.standard_normal((G, n, d))
    h = O.h2o_score(q, k, 1 / math.sqrt(d))
    Hn = _harmonic(n)
    for t in range(n):
        exact = G * (Hn - _harmonic(t))
        assert abs(h[t] - float(exact)) < 1e-12, (t, h[t], float(exact))


def _two_level_prob(z, n_hot, n_cold):
    """Softmax of n_hot logits z and n_cold logits 0: (p_hot, p_cold)."""
    den = n_hot * math.exp(z) + n_cold
    return math.exp(z) / den, 1.0 / den


def pin_two_level_scale(O, rng):
    """Keys c*e0 on a set A and 0 elsewhere, queries x*e0: the logit on A is
    z = x*c/sqrt(d), which fixes the softmax scale 1/sqrt(d)."""
    d, n, W, G = 64, 30, 5, 1
    x, c = 2.0, 2.0
    A = {1, 4, 9, 27, 28}
    k = np.zeros((n, d))
    for t in A:
        k[t, 0] = c
    qw = np.zeros((G, W, d))
    qw[:, :, 0] = x
    z = x * c / math.sqrt(d)
    s = O.snapkv_prepool(qw, k, W, 1 / math.sqrt(d))
    expect = np.zeros(n)
    for p in range(n - W, n):
        n_hot = sum(1 for t in A if t <= p)
        ph, pc = _two_level_prob(z, n_hot, p + 1 - n_hot)
        for t in range(p + 1):
            expect[t] += ph if t in A else pc
    assert np.allclose(s, expect, rtol=1e-12, atol=0)


def pin_window_covering_is_h2o(O, rng):
    """With W >= n every query is in the window, so SnapKV equals H2O."""
    d, G, n = 16, 2, 19
    q = rng.standard_normal((G, n, d))
    k = rng.standard_normal((n, d))
    qw = np.zeros((G, 24, d))
    qw[:, :n, :] = q
    a = O.snapkv_prepool(qw, k, 24, 0.3)
    b = O.h2o_score(q, k, 0.3)
    assert np.allclose(a, b, rtol=1e-12, atol=1e-14)


def pin_gqa_grouping(O, rng):
    """Query heads h*G .. h*G+G-1 share KV head h (grouped-query attention).
    KV head 0 has identical keys (uniform closed form whatever the queries);
    KV head 1 has one hot key at t=0 and its group's queries point at it."""
    L, b, Hq, Hkv, d, n, W = 1, 1, 4, 2, 8, 16, 4
    G = Hq // Hkv
    k = np.zeros((L, b, Hkv, n, d))
    k[0, 0, 0, :, :] = 1.0
    k[0, 0, 1, 0, 0] = 4.0
    qw = np.zeros((L, b, Hq, W, d))
    qw[0, 0, 0:2] = rng.choice([-1.0, 1.0, 2.0], size=(2, W, d))
    qw[0, 0, 2:4, :, 0] = 2.0
    batch = O.Batch(L, b, Hq, Hkv, d, n)
    res = O.snapkv_batch(batch, _bf16_bits(qw), _bf16_bits(k), W, 1, scale=1 / math.sqrt(d))
    s0 = res[0][0]
    for t in range(n):
        exact = G * sum(Fraction(1, p + 1) for p in range(n - W, n) if p >= t)
        assert abs(s0[t] - float(exact)) < 1e-12
    s1 = res[1][0]
    z = 2.0 * 4.0 / math.sqrt(d)
    expect = np.zeros(n)
    for p in range(n - W, n):
        ph, pc = _two_level_prob(z, 1, p)
        expect[0] += G * ph
        expect[1:p + 1] += G * pc
    assert np.allclose(s1, expect, rtol=1e-12, atol=0)


# ---------------------------------------------------------------- pooling ---

def pin_maxpool(O, rng):
    """Hand-worked pools, the k=1 identity, s~ >= s, and scipy's
    maximum_filter1d with -inf padding as an independent routine."""
    g = _golden("maxpool_worked_examples.json")
    s = np.array(g["s"], dtype=np.float64)
    for case in g["cases"]:
        assert np.array_equal(O.maxpool1d(s, case["k"]), np.array(case["out"], dtype=np.float64))
    x = rng.random(101)
    assert np.array_equal(O.maxpool1d(x, 1), x)
    for k in (3, 5, 7, 11, 15):
        y = O.maxpool1d(x, k)
        assert np.all(y >= x)
        ref = maximum_filter1d(x, size=k, mode="constant", cval=-np.inf)
        assert np.array_equal(y, ref)
    short = rng.random(2)
    assert np.array_equal(O.maxpool1d(short, 7), np.full(2, short.max()))


# ---------------------------------------------------------------- budget ----

def pin_kept_count(O, rng):
    g = _golden("quota_worked_examples.json")["kept_count"]
    for n, B, k in g["cases"]:
        assert O.kept_count(n, B) == k, (n, B, O.kept_count(n, B), k)
    for n in (1, 2, 3, 1000, 32768, 100003):
        for B in (0.05, 0.1, 0.2, 0.3, 0.5, 0.75, 1.0):
            k = O.kept_count(n, B)
            exact = Fraction(round(B * 1e6), 10**6) * n
            assert k == math.ceil(exact), (n, B, k)


def pin_quota_golden(O, rng):
    g = _golden("quota_worked_examples.json")
    for ex in g["examples"]:
        q = O.role_quotas(ex["counts"], ex["alpha"], ex["budget"], ex["n"])
        assert q == ex["quotas"], (ex["name"], q, ex["quotas"])
        assert sum(q) == ex["kept"]


def _water_level(counts, weights, K):
    """Independent formulation: the ideal (real-valued) split is
    x_r = min(n_r, w_r * lam) with lam chosen so that sum x_r = K; lam is
    found by walking the breakpoints n_r / w_r in increasing order."""
    live = [r for r in range(len(counts)) if weights[r] > 0 and counts[r] > 0]
    if K == 0 or not live:
        return {r: Fraction(0) for r in live}
    order = sorted(live, key=lambda r: Fraction(counts[r], weights[r]))
    fixed_sum, free_w = 0, sum(weights[r] for r in live)
    for i, r in enumerate(order):
        lam = Fraction(K - fixed_sum, free_w)
        if weights[r] * lam <= counts[r]:
            break
        fixed_sum += counts[r]
        free_w -= weights[r]
    else:
        return {r: Fraction(counts[r]) for r in live}
    return {r: min(Fraction(counts[r]), weights[r] * lam) for r in live}


def pin_quota_waterlevel(O, rng):
    """Quotas sum to K = min(ceil(B n), eligible), never exceed a bucket,
    equal the bucket size where the ideal split saturates it, and otherwise
    lie within one of the exact rational ideal split."""
    for _ in range(400):
        R = int(rng.integers(1, 9))
        counts = [int(x) for x in rng.integers(0, 60, size=R)]
        if rng.random() < 0.3:
            counts[int(rng.integers(R))] = 0
        n = sum(counts)
        if n == 0:
            continue
        alpha = [float(np.float32(x)) for x in rng.choice([0.0, 0.02, 0.05, 0.2, 0.25, 0.7, 0.33], size=R)]
        B = float(rng.choice([0.05, 0.1, 0.2, 0.3, 0.5, 0.9, 1.0]))
        q = O.role_quotas(counts, alpha, B, n)
        w = [round(a * 1e6) for a in alpha]
        elig = sum(c for c, a in zip(counts, w) if a > 0)
        K = min(math.ceil(Fraction(round(B * 1e6), 10**6) * n), elig)
        assert sum(q) == K, (counts, alpha, B, q, K)
        ideal = _water_level(counts, w, K)
        for r in range(R):
            assert 0 <= q[r] <= counts[r]
            if r not in ideal:
                assert q[r] == 0
                continue
            x = ideal[r]
            assert math.floor(x) <= q[r] <= math.ceil(x), (counts, alpha, B, q, r, x)


def pin_key_ban(O, rng):
    """alpha_KEY = 0 keeps no KEY token (the role the method is built to zero,
    Section 4.1 'Hyperparameters'), whatever the scores."""
    b, n, Hkv = 2, 300, 2
    batch = O.Batch(1, b, Hkv * 2, Hkv, 8, n)
    roles = rng.integers(0, 4, size=(b, n)).astype(np.uint8)
    scores = {}
    for u in range(batch.n_units):
        _, s, _ = batch.unit(u)
        sc = rng.random(n)
        sc[roles[s] == 1] += 100.0    # KEY tokens score highest
        scores[u] = sc
    for B in (0.05, 0.2, 0.5, 0.9):
        res = O.select_batch(batch, scores, roles, 4, [0.25, 0.5, 0.70, 0.05], 1, 0.0, B)
        for u, (idx, per_role) in res.items():
            _, s, _ = batch.unit(u)
            kept = idx[idx >= 0]
            assert per_role[1] == 0
            assert np.all(roles[s][kept] != 1)
            elig = int((roles[s] != 1).sum())
            assert kept.size == min(math.ceil(Fraction(round(B * 1e6), 10**6) * n), elig)
            assert np.all(np.diff(kept) > 0)


def pin_global_is_full_sort(O, rng):
    """GLOBAL policy with no ban is plain top-K by score with ties to the
    lower index: numpy's stable argsort of -score, first K, sorted."""
    n = 500
    for trial in range(6):
        sc = rng.integers(0, 40, size=n).astype(np.float64)   # many ties
        roles = rng.integers(0, 4, size=n)
        for B in (0.05, 0.2, 0.5):
            K = O.kept_count(n, B)
            q = O.role_quotas([int((roles == r).sum()) for r in range(4)], [1, 1, 1, 1], B, n,
                              policy=O.POLICY_GLOBAL)
            bk = O.bucket_of_tokens(roles, O.POLICY_GLOBAL, 0)
            idx = O.select_unit(sc, bk, q)
            ref = np.sort(np.argsort(-sc, kind="stable")[:K])
            assert np.array_equal(idx, ref)


def pin_bruteforce_select(O, rng):
    """For tiny units, each bucket's kept set is the subset of its size that
    maximises the score sum, and among those the smallest index tuple
    (exhaustive enumeration, integer scores so sums are exact)."""
    for trial in range(25):
        n = int(rng.integers(6, 15))
        roles = rng.integers(0, 3, size=n)
        sc = rng.integers(0, 5, size=n).astype(np.float64)
        counts = [int((roles == r).sum()) for r in range(3)]
        B = float(rng.choice([0.2, 0.3, 0.5, 0.7]))
        q = O.role_quotas(counts, [0.5, 0.3, 0.2], B, n)
        idx = O.select_unit(sc, roles, q)
        for r in range(3):
            members = [int(t) for t in np.nonzero(roles == r)[0]]
            best = None
            for sub in itertools.combinations(members, q[r]):
                key = (-sum(sc[list(sub)]), sub)
                best = key if best is None or key < best else best
            chosen = tuple(int(t) for t in idx if roles[t] == r)
            assert chosen == best[1], (trial, r, chosen, best)


def pin_compact(O, rng):
    """Compaction is numpy's take on the token axis; -1 gives a zero row."""
    rows = rng.integers(0, 2**16, size=(50, 8)).astype(np.uint16)
    idx = np.array([0, 3, 4, 17, 49, -1, -1])
    out = O.compact_unit(rows, idx)
    assert np.array_equal(out[:5], np.take(rows, idx[:5], axis=0))
    assert np.all(out[5:] == 0)


def pin_varlen_matches_dense(O, rng):
    """The packed (varlen) layout gives the same per-unit scores as the dense
    layout when every sequence has the same length."""
    L, b, Hq, Hkv, d, n, W = 2, 3, 4, 2, 8, 12, 4
    kd = rng.integers(0x3c00, 0x4000, size=(L, b, Hkv, n, d)).astype(np.uint16)
    qd = rng.integers(0x3c00, 0x4000, size=(L, b, Hq, n, d)).astype(np.uint16)
    qw = rng.integers(0x3c00, 0x4000, size=(L, b, Hq, W, d)).astype(np.uint16)
    kv = np.ascontiguousarray(np.transpose(kd, (0, 1, 3, 2, 4)).reshape(L, b * n, Hkv, d))
    qv = np.ascontiguousarray(np.transpose(qd, (0, 1, 3, 2, 4)).reshape(L, b * n, Hq, d))
    dense = O.Batch(L, b, Hq, Hkv, d, n)
    var = O.Batch(L, b, Hq, Hkv, d, n, seqlens=[n] * b)
    a = O.snapkv_batch(dense, qw, kd, W, 3)
    c = O.snapkv_batch(var, qw, kv, W, 3)
    for u in a:
        assert np.array_equal(a[u][1], c[u][1])
    a = O.h2o_batch(dense, qd, kd)
    c = O.h2o_batch(var, qv, kv)
    for u in a:
        assert np.allclose(a[u], c[u], rtol=1e-14, atol=0)


def pin_fair_quotas(O, rng):
    """FAIR (equal retention rate per role, Section 5 'Fair-eviction
    baseline'): the exact rational share of role r is n_r K / N over the
    non-banned roles; the quotas are its floors, and the K - sum(floors) roles
    with the largest fractional parts (ties to the lower role) get one more."""
    for _ in range(300):
        R = int(rng.integers(1, 9))
        counts = [int(x) for x in rng.integers(0, 80, size=R)]
        ban = int(rng.integers(0, 1 << R)) if rng.random() < 0.3 else 0
        n = sum(counts)
        if n == 0:
            continue
        B = float(rng.choice([0.05, 0.1, 0.2, 0.3, 0.5, 1.0]))
        q = O.role_quotas(counts, [0.7] * R, B, n, policy=O.POLICY_FAIR, ban_mask=ban)
        live = [r for r in range(R) if not (ban >> r) & 1 and counts[r] > 0]
        N = sum(counts[r] for r in live)
        K = min(math.ceil(Fraction(round(B * 1e6), 10**6) * n), N)
        assert sum(q) == K
        if N == 0:
            assert q == [0] * R
            continue
        share = {r: Fraction(counts[r] * K, N) for r in live}
        floors = {r: math.floor(share[r]) for r in live}
        extra = K - sum(floors.values())
        up = sorted(live, key=lambda r: (-(share[r] - floors[r]), r))[:extra]
        for r in range(R):
            want = floors[r] + (1 if r in up else 0) if r in share else 0
            assert q[r] == want, (counts, ban, B, q)
    # equal rates exactly when the shares are integers: every role keeps B of its tokens
    q = O.role_quotas([100, 40, 60, 200], [0] * 4, 0.25, 400, policy=O.POLICY_FAIR)
    assert q == [25, 10, 15, 50]


def pin_slack_fill(O, rng):
    """SLACK (unused budget of saturated buckets filled by score): the quotas
    are one round of the alpha split (exact rational shares, floors plus
    largest remainders) capped at each bucket's size; when nothing saturates
    the selection is ROLE_QUOTA's; on tiny units the tokens added beyond the
    per-bucket top-q are the brute-force best subset of the remaining
    eligible tokens, and a role with alpha 0 keeps nothing."""
    for _ in range(300):
        R = int(rng.integers(1, 7))
        counts = [int(x) for x in rng.integers(0, 60, size=R)]
        alpha = [float(x) for x in rng.choice([0.0, 0.02, 0.05, 0.2, 0.25, 0.7], size=R)]
        n = sum(counts)
        if n == 0:
            continue
        B = float(rng.choice([0.05, 0.1, 0.3, 0.5, 1.0]))
        q = O.role_quotas(counts, alpha, B, n, policy=O.POLICY_SLACK)
        a = {r: Fraction(round(alpha[r] * 1e6), 10**6) for r in range(R)}
        E = [r for r in range(R) if a[r] > 0 and counts[r] > 0]
        K = min(math.ceil(Fraction(round(B * 1e6), 10**6) * n), sum(counts[r] for r in E))
        if not E:
            assert q == [0] * R
            continue
        A = sum(a[r] for r in E)
        share = {r: a[r] * K / A for r in E}
        floors = {r: math.floor(share[r]) for r in E}
        up = sorted(E, key=lambda r: (-(share[r] - floors[r]), r))[:K - sum(floors.values())]
        for r in range(R):
            want = min(counts[r], floors[r] + (1 if r in up else 0)) if r in E else 0
            assert q[r] == want, (counts, alpha, B, q)
        assert sum(q) <= K
    # nothing saturates: the same keep set as the proportional split
    b, n = 1, 400
    batch = O.Batch(1, b, 1, 1, 8, n)
    roles = np.repeat(np.arange(4, dtype=np.uint8), 100)[None, :]
    sc = {0: rng.random(n)}
    al = [0.25, 0.25, 0.25, 0.25]
    same_q = O.select_batch(batch, sc, roles, 4, al, -1, 0.0, 0.2, O.POLICY_ROLE_QUOTA)[0][0]
    same_s = O.select_batch(batch, sc, roles, 4, al, -1, 0.0, 0.2, O.POLICY_SLACK)[0][0]
    assert np.array_equal(same_q, same_s)
    for trial in range(30):
        m = int(rng.integers(8, 14))
        tb = O.Batch(1, 1, 1, 1, 8, m)
        rl = rng.integers(0, 3, size=(1, m)).astype(np.uint8)
        rl[0, 0] = 0                                    # role 0 is small: it saturates
        rl[0, 1:] = np.where(rl[0, 1:] == 0, 1, rl[0, 1:])
        sc = rng.integers(0, 5, size=m).astype(np.float64)
        B = float(rng.choice([0.4, 0.5, 0.7]))
        akey = float(rng.choice([0.0, 0.1]))
        al = [0.8, 0.2, 0.0]                            # role 2 is the key role below
        idx, per = O.select_batch(tb, {0: sc}, rl, 3, al, 2, akey, B, O.POLICY_SLACK)[0]
        kept = [int(t) for t in idx if t >= 0]
        counts = [int((rl[0] == x).sum()) for x in range(3)]
        q = O.role_quotas(counts, [0.8, 0.2, akey], B, m, policy=O.POLICY_SLACK)
        E = [x for x in range(3) if counts[x] > 0 and [0.8, 0.2, akey][x] > 0]
        K = min(O.kept_count(m, B), sum(counts[x] for x in E))
        assert len(kept) == K, (trial, kept, K)
        base = set()
        for r in range(3):
            members = [t for t in range(m) if rl[0, t] == r]
            best = min(((-sum(sc[list(sub)]), sub) for sub in itertools.combinations(members, q[r])))
            base |= set(best[1])
        assert base <= set(kept)
        rest = [t for t in range(m) if rl[0, t] in E and t not in base]
        extra = tuple(t for t in kept if t not in base)
        best = min(((-sum(sc[list(sub)]), sub) for sub in itertools.combinations(rest, K - len(base))))
        assert extra == best[1], (trial, extra, best)
        if akey == 0.0:
            assert per[2] == 0


def pin_ceil_quotas(O, rng):
    """CEIL (Algorithm 1's per-bucket ceilings read literally): hand-worked
    quotas; every eligible bucket takes the ceiling of its exact water-level
    share (an independent formulation), so no quota is below the exact
    split's, the total exceeds K by less than the number of unsaturated
    buckets, and the kept set contains the exact split's; rows are padded
    with -1 to min(n, ceil(B n) + kept_extra)."""
    for ex in _golden("ceil_quota_worked_examples.json")["examples"]:
        q = O.role_quotas(ex["counts"], ex["alpha"], ex["budget"], ex["n"], policy=O.POLICY_CEIL)
        assert q == ex["quotas"], (ex["name"], q, ex["quotas"])
        assert sum(q) == ex["kept"]
    for _ in range(400):
        R = int(rng.integers(1, 9))
        counts = [int(x) for x in rng.integers(0, 60, size=R)]
        n = sum(counts)
        if n == 0:
            continue
        alpha = [float(np.float32(x)) for x in rng.choice([0.0, 0.02, 0.05, 0.2, 0.25, 0.7, 0.33], size=R)]
        B = float(rng.choice([0.05, 0.1, 0.2, 0.3, 0.5, 0.9, 1.0]))
        q = O.role_quotas(counts, alpha, B, n, policy=O.POLICY_CEIL)
        q0 = O.role_quotas(counts, alpha, B, n)
        w = [round(a * 1e6) for a in alpha]
        elig = sum(c for c, a in zip(counts, w) if a > 0)
        K = min(math.ceil(Fraction(round(B * 1e6), 10**6) * n), elig)
        ideal = _water_level(counts, w, K)
        for r in range(R):
            assert q[r] == (math.ceil(ideal[r]) if r in ideal else 0), (counts, alpha, B, q, r)
            assert q0[r] <= q[r] <= counts[r]
        unsat = sum(1 for r in ideal if ideal[r] < counts[r])
        assert K <= sum(q) <= K + max(unsat - 1, 0), (counts, alpha, B, q, K)
    b, n = 2, 500
    for extra in (3, 7):
        batch = O.Batch(1, b, 2, 1, 8, n, kept_extra=extra)
        roles = rng.integers(0, 4, size=(b, n)).astype(np.uint8)
        sc = {u: rng.random(n) for u in range(b)}
        al = [0.25, 0.02, 0.70, 0.05]
        for B, keep_last in ((0.05, 0), (0.13, 0), (0.3, 16), (0.999, 0)):
            ceil_sel = O.select_batch(batch, sc, roles, 4, al, -1, 0.0, B, O.POLICY_CEIL, keep_last=keep_last)
            exact_sel = O.select_batch(batch, sc, roles, 4, al, -1, 0.0, B, keep_last=keep_last)
            width = min(n, math.ceil(Fraction(round(B * 1e6), 10**6) * n) + extra)
            for u in range(b):
                idx, per = ceil_sel[u]
                assert idx.shape == (width,)
                kept = idx[idx >= 0]
                assert np.all(idx[kept.size:] == -1) and np.all(np.diff(kept) > 0)
                assert set(exact_sel[u][0][exact_sel[u][0] >= 0]) <= set(kept)
                assert sum(per) == kept.size
                assert np.all(kept[kept.size - keep_last:] == np.arange(n - keep_last, n)) if keep_last else True


def pin_recency_floor(O, rng):
    """The recency floor keeps the last R = min(keep_last, n, ceil(B n))
    tokens and splits the other ceil(B n) - R slots over the earlier tokens:
    keep_last = 0 is the plain selection, a floor as large as the budget keeps
    exactly the last ceil(B n) tokens, and on tiny units each bucket's kept
    subset of the prefix is the brute-force best of its size."""
    b, n = 2, 240
    batch = O.Batch(1, b, 2, 1, 8, n)
    roles = rng.integers(0, 4, size=(b, n)).astype(np.uint8)
    scores = {u: rng.random(n) for u in range(batch.n_units)}
    al = [0.25, 0.02, 0.70, 0.05]
    for B in (0.05, 0.3):
        plain = O.select_batch(batch, scores, roles, 4, al, 1, 0.02, B)
        zero = O.select_batch(batch, scores, roles, 4, al, 1, 0.02, B, keep_last=0)
        K = O.kept_count(n, B)
        full = O.select_batch(batch, scores, roles, 4, al, 1, 0.02, B, keep_last=10 * n)
        for u in plain:
            assert np.array_equal(plain[u][0], zero[u][0])
            assert np.array_equal(full[u][0], np.arange(n - K, n))
    for trial in range(30):
        m = int(rng.integers(8, 15))
        tb = O.Batch(1, 1, 1, 1, 8, m)
        rl = rng.integers(0, 3, size=(1, m)).astype(np.uint8)
        sc = rng.integers(0, 5, size=m).astype(np.float64)
        B = float(rng.choice([0.3, 0.5, 0.7]))
        keep = int(rng.integers(1, 4))
        idx, per = O.select_batch(tb, {0: sc}, rl, 3, [0.5, 0.3, 0.2], -1, 0.0, B, keep_last=keep)[0]
        K = O.kept_count(m, B)
        R = min(keep, m, K)
        kept = [int(t) for t in idx if t >= 0]
        assert len(kept) == K
        assert kept[-R:] == list(range(m - R, m))
        prefix = [t for t in kept if t < m - R]
        for r in range(3):
            members = [t for t in range(m - R) if rl[0, t] == r]
            chosen = tuple(t for t in prefix if rl[0, t] == r)
            best = min(((-sum(sc[list(sub)]), sub) for sub in itertools.combinations(members, len(chosen))))
            assert chosen == best[1], (trial, r, chosen, best)
        assert per == [int((rl[0, kept] == x).sum()) for x in range(3)]


def pin_quest_bound(O, rng):
    """Quest page bound: with one-token pages it is the plain dot product of
    the mean window query with each key; for any page it is at least every
    member's dot product, reaches it when the page's keys are equal, does not
    depend on the order of tokens inside a page, and the mean query is the
    plain average of the G x W_eff window rows."""
    G, W, d, n = 3, 5, 6, 37
    qw = rng.standard_normal((G, W, d))
    k = rng.standard_normal((n, d))
    qbar = qw.reshape(-1, d).mean(axis=0)
    assert np.allclose(O.quest_score(qw, k, W, 1), k @ qbar, rtol=1e-12, atol=1e-12)
    for page in (2, 4, 16):
        u = O.quest_score(qw, k, W, page)
        dots = k @ qbar
        for p0 in range(0, n, page):
            assert np.all(u[p0:p0 + page] == u[p0])
            assert u[p0] >= dots[p0:p0 + page].max() - 1e-12
        perm = k.copy()
        for p0 in range(0, n, page):
            blk = perm[p0:p0 + page]
            perm[p0:p0 + page] = blk[rng.permutation(blk.shape[0])]
        assert np.allclose(O.quest_score(qw, perm, W, page), u, rtol=0, atol=1e-12)
    same = np.repeat(rng.standard_normal((1, d)), 8, axis=0)
    assert np.allclose(O.quest_score(qw, same, W, 8), same @ qbar, rtol=1e-12, atol=1e-12)
    # a window longer than the sequence uses every position (W_eff = n)
    short = rng.standard_normal((3, d))
    qbar3 = qw[:, :3].reshape(-1, d).mean(axis=0)
    assert np.allclose(O.quest_score(qw, short, W, 1), short @ qbar3, rtol=1e-12, atol=1e-12)
    # hand-worked pages where the per-dimension bound lies strictly above the
    # page's best dot product (so an exact per-page maximum would fail here)
    g = _golden("quest_bound_worked_examples.json")
    qg = np.asarray(g["q_win"], dtype=np.float64)
    for case in g["cases"]:
        keys = np.asarray(case["keys"], dtype=np.float64)
        got = O.quest_score(qg, keys, g["W"], case["page"])
        assert np.array_equal(got, np.asarray(case["bound"], dtype=np.float64)), (case, got)


def pin_decode_attention(O, rng):
    """Decode attention: equal keys give the plain mean of the value rows; one
    key far above the rest gives (nearly) its value row; the output is a
    convex combination (inside the per-dim range of the values); row order
    does not matter; rows flagged invalid are ignored whatever they hold; an
    empty cache gives zero."""
    G, m, d = 3, 20, 8
    q = rng.standard_normal((G, d))
    v = rng.standard_normal((m, d))
    kc = np.repeat(rng.standard_normal((1, d)), m, axis=0)
    ok = np.ones(m, dtype=bool)
    assert np.allclose(O.decode_attention(q, kc, v, ok, 0.3), np.tile(v.mean(axis=0), (G, 1)),
                       rtol=0, atol=1e-12)
    k = rng.standard_normal((m, d))
    k[7] = 50.0 * q[0] / np.linalg.norm(q[0])
    o = O.decode_attention(q[:1], k, v, ok, 1.0)
    assert np.allclose(o[0], v[7], atol=1e-6)
    o = O.decode_attention(q, k, v, ok, 0.5)
    assert np.all(o >= v.min(axis=0) - 1e-12) and np.all(o <= v.max(axis=0) + 1e-12)
    perm = rng.permutation(m)
    assert np.allclose(O.decode_attention(q, k[perm], v[perm], ok, 0.5), o, rtol=1e-12, atol=1e-12)
    junk_k = np.vstack([k, 1e3 * rng.standard_normal((5, d))])
    junk_v = np.vstack([v, 1e3 * rng.standard_normal((5, d))])
    flags = np.concatenate([ok, np.zeros(5, dtype=bool)])
    assert np.allclose(O.decode_attention(q, junk_k, junk_v, flags, 0.5), o, rtol=1e-12, atol=1e-12)
    assert np.all(O.decode_attention(q, k, v, np.zeros(m, dtype=bool), 0.5) == 0)
    # closed form at a scale other than 1: two keys 4 e_0 ("hot") and two zero
    # keys, values 8 e_j.  With scale 1/4 a query (ln 3, ...) gives the hot
    # keys logit ln 3 and the cold ones 0, so the weights are 3/8, 3/8, 1/8,
    # 1/8 and the output (3, 3, 1, 1); a query (-ln 3, ...) gives weights
    # 1/8, 1/8, 3/8, 3/8 and the output (1, 1, 3, 3).  Components of q along
    # dimensions where every key is 0 do not matter.
    ln3 = math.log(3.0)
    qs = np.array([[ln3, 0.0, 0.0, 0.0], [-ln3, 0.7, -1.1, 0.3]])
    ks = np.array([[4.0, 0, 0, 0], [4.0, 0, 0, 0], [0.0, 0, 0, 0], [0.0, 0, 0, 0]])
    vs = 8.0 * np.eye(4)
    want = np.array([[3.0, 3.0, 1.0, 1.0], [1.0, 1.0, 3.0, 3.0]])
    got = O.decode_attention(qs, ks, vs, np.ones(4, dtype=bool), 0.25)
    assert np.allclose(got, want, rtol=0, atol=1e-12), got


ALL_PINS = [
    pin_rows_sum_to_one, pin_snapkv_total, pin_h2o_total, pin_uniform_closed_forms,
    pin_two_level_scale, pin_window_covering_is_h2o, pin_gqa_grouping, pin_maxpool,
    pin_kept_count, pin_quota_golden, pin_quota_waterlevel, pin_key_ban,
    pin_global_is_full_sort, pin_bruteforce_select, pin_compact, pin_varlen_matches_dense,
    pin_fair_quotas, pin_recency_floor, pin_quest_bound, pin_decode_attention, pin_slack_fill,
    pin_ceil_quotas,
]
