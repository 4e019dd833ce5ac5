"""Reference oracle for role-conditional KV-cache eviction (arXiv 2607.13205).

TEST INFRASTRUCTURE ONLY.  This module is the slow, plain, fp64 statement of
what the GPU library computes.  Only ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py`` may import it; the library itself
never does, and it shares no code with the CUDA path (the two meet only in
the seeded input generator, which holds none of the method's arithmetic).

Everything is computed from the definitions, in float64, with numpy's
matmul / sort as the only library steps:

* ``attention_probs``   -- softmax probabilities p_t(q) of the causal prefill
                           attention (the quantity both scores sum; Section 2).
* ``snapkv_prepool``    -- SnapKV windowed mass: sum of p_t(q) over the last W
                           queries, GQA query heads of a KV head summed
                           (Section 2; Section 4 "SnapKV mechanism";
                           Algorithm 1, the windowed-mass step).
* ``h2o_score``         -- H2O accumulated mass s(t) = sum_q p_t(q) over every
                           causal query (Section 2).
* ``quest_score``       -- the one-shot Quest analogue: page key-bounds against
                           the window's mean query (Section 5, "Query-aware
                           baseline").
* ``decode_attention``  -- one decode step of attention through the compacted
                           cache (Section 6).
* ``maxpool1d``         -- the 1-D max-pool along the KV axis
                           (Algorithm 1, the pooling step; Section 4).
* ``kept_count``,
  ``role_quotas``       -- the per-role budget split of the combined method:
                           top-ceil(alpha_r B n_kv) per role bucket, alpha
                           renormalised over buckets, slack from saturated
                           buckets redistributed (Section 4.1; Algorithm 1).
                           Four more splits: GLOBAL (plain top-k, optional
                           role ban; Sections 2 and 4), FAIR (equal
                           retention rate per role; Section 5
                           "Fair-eviction baseline"), SLACK (the slack of
                           saturated buckets filled by score instead of
                           in proportion to alpha) and CEIL (Algorithm 1's
                           per-bucket ceilings taken literally, so the
                           total may exceed ceil(B n)).
* ``select_unit``       -- per-bucket top-q_r by pooled score (Algorithm 1);
                           ``select_batch`` optionally keeps the last R
                           tokens first (SnapKV's recency floor, Section 7).
* ``compact_unit``      -- gather of the kept K/V rows into a dense cache
                           (Section 6 "Systems cost": the compacting
                           implementation the paper describes but does not
                           build).

Readings of points the paper leaves open (all listed in the design notes):
softmax scale 1/sqrt(d); causal masking inside the window; window = the last
W_eff = min(W, n) positions; GQA heads are summed, not averaged; the pool is
stride 1, same length, truncated at the sequence edges; "renormalized per
bucket" = alpha_r / sum of alpha over the eligible buckets (alpha_r > 0 and
n_r > 0) of the sequence; the total kept is exactly ceil(B n) (or all
eligible tokens when fewer), apportioned by integer water-filling plus
largest remainder (the CEIL split alone takes Algorithm 1's ceilings
literally and may keep a few more); ties in score go to the lower token index; kept indices
are returned in ascending position order.  Budgets and alphas are taken to
fixed point with six decimals so that ceilings are exact.
"""

from __future__ import annotations

import math
from typing import Iterable, Sequence

import numpy as np

FIXED_ONE = 1_000_000  # fixed-point unit for budgets and alphas (6 decimals)

POLICY_ROLE_QUOTA = 0
POLICY_GLOBAL = 1
POLICY_FAIR = 2
POLICY_SLACK = 3
POLICY_CEIL = 4


# ----------------------------------------------------------------------------
# conversions
# ----------------------------------------------------------------------------

def bf16_to_f64(bits) -> np.ndarray:
    """bfloat16 bit patterns (uint16) -> float64, exactly."""
    b = np.asarray(bits).astype(np.uint16, copy=False)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def to_fixed(x: float) -> int:
    """Round a float32 parameter (budget or alpha) to an integer count of
    1e-6 units, half away from zero: floor(double(x) * 1e6 + 0.5)."""
    v = float(np.float32(x))
    if not math.isfinite(v) or v < 0:
        raise ValueError(f"parameter must be finite and >= 0, got {x!r}")
    return int(math.floor(v * 1e6 + 0.5))


# ----------------------------------------------------------------------------
# attention probabilities and the two scores (Section 2, Section 4)
# ----------------------------------------------------------------------------

def attention_probs(q_rows: np.ndarray, k: np.ndarray, positions: np.ndarray,
                    scale: float) -> np.ndarray:
    """Softmax probabilities of causal attention.

    q_rows: (R, d) query vectors; positions: (R,) their token positions;
    k: (n, d) keys.  Row r attends to keys t <= positions[r] with logits
    scale * <q_r, k_t>; returns P with P[r, t] = p_t(q_r) (zero where masked).
    The row softmax is the plain definition: subtract the row max, exponentiate,
    divide by the row sum.
    """
    q_rows = np.asarray(q_rows, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    n = k.shape[0]
    logits = scale * (q_rows @ k.T)                       # (R, n)
    visible = np.arange(n)[None, :] <= np.asarray(positions)[:, None]
    logits = np.where(visible, logits, -np.inf)
    m = logits.max(axis=1, keepdims=True)
    e = np.where(visible, np.exp(logits - m), 0.0)
    return e / e.sum(axis=1, keepdims=True)


def window_positions(n: int, W: int) -> np.ndarray:
    """Positions of the SnapKV observation window: the last W_eff = min(W, n)
    queries of the sequence (Section 4, 'SnapKV mechanism')."""
    w_eff = min(W, n)
    return np.arange(n - w_eff, n)


def snapkv_prepool(q_win: np.ndarray, k: np.ndarray, W: int, scale: float) -> np.ndarray:
    """SnapKV windowed mass before pooling, for one (layer, sequence, KV head).

    q_win: (G, W, d) -- the window queries of the G query heads that share this
    KV head; row i of each head sits at position n - W_eff + i, rows
    i >= W_eff are ignored.  k: (n, d).
    s(t) = sum over heads g and window rows i of p_t(q_{g,i})  (Algorithm 1,
    windowed mass; GQA heads summed).
    """
    n = k.shape[0]
    G = q_win.shape[0]
    w_eff = min(W, n)
    if n == 0:
        return np.zeros(0)
    pos = window_positions(n, W)
    s = np.zeros(n)
    for g in range(G):
        P = attention_probs(q_win[g, :w_eff, :], k, pos, scale)
        s += P.sum(axis=0)
    return s


def h2o_score(q: np.ndarray, k: np.ndarray, scale: float, row_block: int = 2048) -> np.ndarray:
    """H2O accumulated mass s(t) = sum_q p_t(q) over every causal prefill
    query q of the G query heads sharing this KV head (Section 2).

    q: (G, n, d) all queries; k: (n, d).  Rows are processed in blocks only to
    bound memory; each block is the same plain softmax.
    """
    G, n, _ = q.shape
    s = np.zeros(n)
    for g in range(G):
        for r0 in range(0, n, row_block):
            r1 = min(n, r0 + row_block)
            P = attention_probs(q[g, r0:r1, :], k, np.arange(r0, r1), scale)
            s += P.sum(axis=0)
    return s


def quest_score(q_win: np.ndarray, k: np.ndarray, W: int, page: int) -> np.ndarray:
    """Quest one-shot analogue (Section 5, "Query-aware baseline"): the mean
    query qbar of the window rows (the last W_eff = min(W, n) positions of all
    G query heads of the KV head) scores every page of `page` consecutive
    keys by Quest's key-bound, sum_i max(qbar_i * min_t k_ti, qbar_i *
    max_t k_ti) over the page's tokens t, an upper bound on qbar . k_t for
    every token of the page; every token gets its page's bound.  The last
    page of a sequence may be short.  q_win is (G, W, d), k is (n, d)."""
    k = np.asarray(k, dtype=np.float64)
    n = k.shape[0]
    out = np.zeros(n)
    if n == 0:
        return out
    w_eff = min(W, n)
    q = np.asarray(q_win, dtype=np.float64)[:, :w_eff, :]
    qbar = q.reshape(-1, q.shape[-1]).mean(axis=0)
    for p0 in range(0, n, page):
        blk = k[p0:p0 + page]
        lo, hi = blk.min(axis=0), blk.max(axis=0)
        out[p0:p0 + page] = np.maximum(qbar * lo, qbar * hi).sum()
    return out


def decode_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, valid: np.ndarray,
                     scale: float) -> np.ndarray:
    """One decode step through a (compacted) cache: each of the G query rows
    q (G, d) attends to the cache rows k, v (m, d) whose `valid` flag is set
    (kept slots; the -1 padding of an infeasible budget is not), o_g =
    sum_j softmax_j(scale q_g . k_j) v_j.  This is the step the compacted
    cache exists for (Section 6: the 1-B memory and latency the masking
    harness does not realise).  Returns (G, d); rows with no valid key give 0."""
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    valid = np.asarray(valid, dtype=bool)
    out = np.zeros((q.shape[0], v.shape[1]))
    if not valid.any():
        return out
    kk, vv = k[valid], v[valid]
    logits = scale * (q @ kk.T)
    m = logits.max(axis=1, keepdims=True)
    e = np.exp(logits - m)
    return (e / e.sum(axis=1, keepdims=True)) @ vv


def maxpool1d(s: np.ndarray, kernel: int) -> np.ndarray:
    """1-D max-pool along the KV axis, stride 1, output the same length,
    window truncated at the sequence edges:
    out(t) = max over |delta| <= kernel//2, 0 <= t+delta < n, of s(t+delta)
    (Algorithm 1, pooling step)."""
    if kernel < 1 or kernel % 2 == 0:
        raise ValueError("pool kernel must be odd and >= 1")
    s = np.asarray(s, dtype=np.float64)
    n = s.shape[0]
    h = kernel // 2
    out = np.empty(n)
    for t in range(n):
        out[t] = s[max(0, t - h): min(n, t + h + 1)].max()
    return out


# ----------------------------------------------------------------------------
# budget split across role buckets (Section 4.1, Algorithm 1)
# ----------------------------------------------------------------------------

def kept_count(n: int, budget: float) -> int:
    """Retained tokens of an n-token sequence at budget B: ceil(B * n), with B
    in fixed point so the ceiling is exact."""
    b = to_fixed(budget)
    if b <= 0 or b > FIXED_ONE:
        raise ValueError("budget must lie in (0, 1]")
    return (b * n + FIXED_ONE - 1) // FIXED_ONE


def role_quotas(counts: Sequence[int], alpha: Sequence[float], budget: float, n: int,
                policy: int = POLICY_ROLE_QUOTA, ban_mask: int = 0,
                k_full: int | None = None) -> list[int]:
    """Per-bucket keep counts q_r for one sequence.

    ROLE_QUOTA (the combined method, Section 4.1): bucket r gets the share
    alpha_r / sum(alpha over eligible buckets) of the budget K, where a bucket
    is eligible when alpha_r > 0, it holds tokens, and it is not banned.
    K = min(ceil(B n), eligible tokens).  A bucket whose share reaches its
    size keeps all its tokens and its unused share goes to the others in
    proportion to their alpha (repeated until no bucket saturates); the rest
    is split by integer floor plus largest remainder (ties to the lower role
    id), so the quotas sum to K exactly.

    GLOBAL (plain H2O / SnapKV top-k, Section 2; the 'No-X' role ban of
    Section 4 when ban_mask is set): one bucket holding every non-banned
    token; its quota is min(ceil(B n), size) and is reported on bucket 0.

    FAIR (the fair-eviction baseline of Section 5, "Fair-eviction baseline":
    equal retention rate per role): as ROLE_QUOTA with the weight of every
    non-banned role equal to its token count, so each role keeps the same
    fraction of its tokens up to integer rounding; alpha is not used.

    SLACK (the other reading of Algorithm 1's "redistribute unused budget
    from saturated buckets"): one round of the ROLE_QUOTA split without the
    water-filling, each quota capped at its bucket's size; the quotas then
    sum to K minus the slack that saturated buckets leave, and select_batch
    fills that slack with the best-scoring remaining tokens of the eligible
    buckets.

    CEIL (Algorithm 1 read literally: bucket r keeps the top
    ceil(alpha_r B n_kv) of its tokens, alpha renormalised over the eligible
    buckets): the ROLE_QUOTA water-filling of saturated buckets, then every
    unsaturated bucket takes the ceiling of its share instead of floor plus
    largest remainder.  Each ceiling exceeds its share by less than one, so
    the quotas sum to between K and K + (unsaturated buckets - 1); the rows
    that hold them must be that much wider than ceil(B n) (Batch.kept_extra).

    k_full, when given, replaces ceil(B n) as the budget to split (the
    recency floor of select_batch takes its tokens out of it first).
    """
    R = len(counts)
    counts = [int(c) for c in counts]
    if k_full is not None:
        K_full = int(k_full)
    else:
        K_full = kept_count(n, budget) if n > 0 else 0
    q = [0] * R
    if policy == POLICY_GLOBAL:
        eligible = sum(counts[r] for r in range(R) if not (ban_mask >> r) & 1)
        q[0] = min(K_full, eligible)
        return q
    if policy == POLICY_FAIR:
        a = [0 if (ban_mask >> r) & 1 else counts[r] for r in range(R)]
    else:
        a = [0 if (ban_mask >> r) & 1 else to_fixed(alpha[r]) for r in range(R)]
    S = [r for r in range(R) if a[r] > 0 and counts[r] > 0]
    K = min(K_full, sum(counts[r] for r in S))
    k_left = K
    while S and policy != POLICY_SLACK:
        A = sum(a[r] for r in S)
        saturated = [r for r in S if a[r] * k_left >= counts[r] * A]
        if not saturated:
            break
        for r in saturated:
            q[r] = counts[r]
            k_left -= counts[r]
        S = [r for r in S if r not in saturated]
    if S and policy == POLICY_CEIL:
        A = sum(a[r] for r in S)
        for r in S:
            q[r] = -((-a[r] * k_left) // A)          # ceil(a_r k_left / A)
    elif S:
        A = sum(a[r] for r in S)
        rem = {}
        for r in S:
            q[r] = (a[r] * k_left) // A
            rem[r] = (a[r] * k_left) % A
        left = k_left - sum(q[r] for r in S)
        for r in sorted(S, key=lambda r: (-rem[r], r))[:left]:
            q[r] += 1
    if policy == POLICY_SLACK:
        q = [min(q[r], counts[r]) for r in range(R)]
    return q


def eligible_roles(counts: Sequence[int], alpha: Sequence[float], policy: int,
                   ban_mask: int) -> list[int]:
    """Roles whose bucket takes part in the split: not banned, holding tokens
    and, for the alpha-weighted policies, alpha_r > 0."""
    R = len(counts)
    return [r for r in range(R) if counts[r] > 0 and not (ban_mask >> r) & 1
            and (policy in (POLICY_GLOBAL, POLICY_FAIR) or to_fixed(alpha[r]) > 0)]


def bucket_of_tokens(roles: np.ndarray, policy: int, ban_mask: int) -> np.ndarray:
    """Bucket id of every token: its role (ROLE_QUOTA, FAIR) or 0 (GLOBAL);
    -1 for tokens of a banned role."""
    roles = np.asarray(roles).astype(np.int64)
    banned = ((ban_mask >> roles) & 1).astype(bool)
    b = np.zeros_like(roles) if policy == POLICY_GLOBAL else roles.copy()
    b[banned] = -1
    return b


def select_unit(scores: np.ndarray, buckets: np.ndarray, quotas: Sequence[int]) -> np.ndarray:
    """Per-bucket top-q_r by score, ties to the lower token index; returns the
    union of kept token indices in ascending order (Algorithm 1, per-role
    top-k and keep-mask)."""
    scores = np.asarray(scores, dtype=np.float64)
    kept = []
    for r, qr in enumerate(quotas):
        if qr <= 0:
            continue
        idx = np.nonzero(buckets == r)[0]
        order = np.lexsort((idx, -scores[idx]))   # score descending, index ascending
        kept.append(idx[order[:qr]])
    if not kept:
        return np.zeros(0, dtype=np.int64)
    return np.sort(np.concatenate(kept))


def compact_unit(rows: np.ndarray, idx: np.ndarray) -> np.ndarray:
    """Dense compressed cache for one unit: out[j] = rows[idx[j]]; a padding
    index (-1) yields a zero row (Section 6, compacting implementation)."""
    idx = np.asarray(idx)
    out = np.zeros((idx.shape[0],) + rows.shape[1:], dtype=rows.dtype)
    ok = idx >= 0
    out[ok] = rows[idx[ok]]
    return out


# ----------------------------------------------------------------------------
# batch drivers over (layer, sequence, KV head) units
# ----------------------------------------------------------------------------

class Batch:
    """Shapes of one call.  Dense layout: K/V [L][b][Hkv][n_max][d],
    queries [L][b][Hq][n_max][d], scores [L][b][Hkv][n_max], roles [b][n_max].
    Varlen layout (seqlens given): K/V [L][T][Hkv][d], queries [L][T][Hq][d],
    scores [L][Hkv][T], roles [T], sequence s occupying tokens
    cu[s] .. cu[s+1]-1.  The SnapKV window queries are always
    [L][b][Hq][W][d]."""

    def __init__(self, L: int, b: int, Hq: int, Hkv: int, d: int, n_max: int,
                 seqlens: Iterable[int] | None = None, kept_extra: int = 0):
        self.L, self.b, self.Hq, self.Hkv, self.d, self.n_max = L, b, Hq, Hkv, d, n_max
        self.kept_extra = int(kept_extra)
        if Hq % Hkv:
            raise ValueError("Hq must be a multiple of Hkv")
        self.G = Hq // Hkv
        self.varlen = seqlens is not None
        self.seqlens = [int(x) for x in seqlens] if seqlens is not None else [n_max] * b
        self.cu = np.concatenate([[0], np.cumsum(self.seqlens)]).astype(np.int64)
        self.T = int(self.cu[-1])

    @property
    def n_units(self) -> int:
        return self.L * self.b * self.Hkv

    def unit(self, u: int) -> tuple[int, int, int]:
        l, rest = divmod(u, self.b * self.Hkv)
        s, h = divmod(rest, self.Hkv)
        return l, s, h

    def kv_rows(self, kv: np.ndarray, u: int) -> np.ndarray:
        l, s, h = self.unit(u)
        n = self.seqlens[s]
        if self.varlen:
            return kv[l, self.cu[s]:self.cu[s] + n, h, :]
        return kv[l, s, h, :n, :]

    def q_rows(self, q: np.ndarray, u: int) -> np.ndarray:
        """(G, n, d) queries of the G heads of KV head h (H2O)."""
        l, s, h = self.unit(u)
        n = self.seqlens[s]
        hs = slice(h * self.G, (h + 1) * self.G)
        if self.varlen:
            return np.transpose(q[l, self.cu[s]:self.cu[s] + n, hs, :], (1, 0, 2))
        return q[l, s, hs, :n, :]

    def roles(self, roles: np.ndarray, s: int) -> np.ndarray:
        n = self.seqlens[s]
        if self.varlen:
            return roles[self.cu[s]:self.cu[s] + n]
        return roles[s, :n]

    def score_view(self, scores: np.ndarray, u: int) -> np.ndarray:
        l, s, h = self.unit(u)
        n = self.seqlens[s]
        if self.varlen:
            return scores[l, h, self.cu[s]:self.cu[s] + n]
        return scores[l, s, h, :n]

    def kept_rows(self, n: int, budget: float) -> int:
        """Width of an n-token sequence's kept row: ceil(B n) slots plus
        kept_extra (room for the CEIL split's overshoot), at most n."""
        return min(n, kept_count(n, budget) + self.kept_extra) if n > 0 else 0

    def kept_offsets(self, budget: float) -> np.ndarray:
        ks = [self.kept_rows(n, budget) for n in self.seqlens]
        return np.concatenate([[0], np.cumsum(ks)]).astype(np.int64)


def snapkv_batch(batch: Batch, q_win_bits, k_bits, W: int, pool_k: int,
                 scale: float | None = None, units: Iterable[int] | None = None):
    """SnapKV scores for the requested units (default: all).  Returns
    {unit: (prepool, pooled)} as float64 arrays of length n_s."""
    scale = 1.0 / math.sqrt(batch.d) if scale is None or scale <= 0 else scale
    out = {}
    for u in (range(batch.n_units) if units is None else units):
        l, s, h = batch.unit(u)
        k = bf16_to_f64(batch.kv_rows(k_bits, u))
        qw = bf16_to_f64(q_win_bits[l, s, h * batch.G:(h + 1) * batch.G, :, :])
        pre = snapkv_prepool(qw, k, W, scale)
        out[u] = (pre, maxpool1d(pre, pool_k) if pre.size else pre)
    return out


def quest_batch(batch: Batch, q_win_bits, k_bits, W: int, page: int, units: Iterable[int] | None = None):
    """quest_score for every unit: {unit: per-token page bound}."""
    out = {}
    for u in (range(batch.n_units) if units is None else units):
        l, s, h = batch.unit(u)
        k = bf16_to_f64(batch.kv_rows(k_bits, u))
        qw = bf16_to_f64(q_win_bits[l, s, h * batch.G:(h + 1) * batch.G])
        out[u] = quest_score(qw, k, W, page)
    return out


def h2o_batch(batch: Batch, q_bits, k_bits, scale: float | None = None,
              units: Iterable[int] | None = None):
    """H2O scores {unit: s} (float64, length n_s) for the requested units."""
    scale = 1.0 / math.sqrt(batch.d) if scale is None or scale <= 0 else scale
    out = {}
    for u in (range(batch.n_units) if units is None else units):
        k = bf16_to_f64(batch.kv_rows(k_bits, u))
        q = bf16_to_f64(batch.q_rows(q_bits, u))
        out[u] = h2o_score(q, k, scale)
    return out


def select_batch(batch: Batch, unit_scores: dict, roles, n_roles: int, alpha: Sequence[float],
                 key_role: int, alpha_key: float, budget: float,
                 policy: int = POLICY_ROLE_QUOTA, ban_mask: int = 0, keep_last: int = 0):
    """Role-conditional selection for each unit in ``unit_scores``.

    alpha[key_role] is replaced by alpha_key (the method's one tuned knob,
    Section 4.1).  keep_last > 0 adds a recency floor (SnapKV's observation
    window, the part of SnapKV Section 7 finds is not what helps): the last
    R = min(keep_last, n, ceil(B n)) tokens are kept whatever their score and
    role, and the remaining ceil(B n) - R slots are split over the earlier
    tokens exactly as without the floor (roles counted over those tokens
    only).  Returns {unit: (kept_idx padded with -1 to the row width
    batch.kept_rows(n, B), kept count per role)}.
    """
    al = [float(np.float32(a)) for a in alpha[:n_roles]]
    if 0 <= key_role < n_roles:
        al[key_role] = float(np.float32(alpha_key))
    out = {}
    for u, sc in unit_scores.items():
        _, s, _ = batch.unit(u)
        r = np.asarray(batch.roles(roles, s)).astype(np.int64)
        n = r.shape[0]
        budget_n = kept_count(n, budget) if n > 0 else 0
        width = batch.kept_rows(n, budget)
        forced = min(int(keep_last), n, budget_n)
        nf = n - forced                              # tokens before the floor
        counts = [int((r[:nf] == x).sum()) for x in range(n_roles)]
        q = role_quotas(counts, al, budget, n, policy, ban_mask, k_full=budget_n - forced)
        bk = bucket_of_tokens(r, policy, ban_mask)
        bk[nf:] = -1
        idx = select_unit(np.asarray(sc, dtype=np.float64), bk, q)
        if policy == POLICY_SLACK:
            # the slack of saturated buckets goes to the best-scoring tokens
            # of eligible buckets not kept yet (ties to the lower index)
            E = eligible_roles(counts, al, policy, ban_mask)
            K = min(budget_n - forced, sum(counts[x] for x in E))
            slack = K - sum(q)
            if slack > 0:
                sc64 = np.asarray(sc, dtype=np.float64)
                pool = np.nonzero(np.isin(r[:nf], E))[0]
                pool = np.setdiff1d(pool, idx)
                order = np.lexsort((pool, -sc64[pool]))
                idx = np.concatenate([idx, pool[order[:slack]]])
        idx = np.sort(np.concatenate([idx, np.arange(nf, n, dtype=np.int64)]))
        padded = np.full(width, -1, dtype=np.int64)
        padded[:idx.shape[0]] = idx
        per_role = [int((r[idx] == x).sum()) for x in range(n_roles)]
        out[u] = (padded, per_role)
    return out
