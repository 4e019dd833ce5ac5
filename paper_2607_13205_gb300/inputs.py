"""Seeded synthetic inputs shaped like the paper's schema-dense workloads.

This module only *makes data*: role streams from a seeded nested-JSON emitter
and bf16 Q/K/V with a role-dependent key structure.  It holds none of the
method's arithmetic and is shared, as an input source, by the tests, the
benchmark and the oracle checks.

Stand-ins (the paper's corpora and models are not available):

* roles: a nested-JSON emitter -- an instruction prefix (OTHER), objects made
  of '{' / ',' / ':' / '}' and indentation (SINK = delimiter + whitespace),
  KEY runs and VALUE runs, nested to a maximum depth with fan-out 2..6, then a
  question suffix (OTHER) that holds the SnapKV window.  Run lengths are set
  so that the shallow corpora have KEY near 42% of tokens (the JSON key
  density of Section 5, 'Role-density boundary') and the deep corpus has
  KEY:VALUE near 1:1 with SINK near 40%.
* keys: K_t = z_t + a u (SINK) + b u (KEY), queries Q = z + c u, values V = z,
  with z ~ N(0,1) per element and u a seeded unit direction per
  (layer, KV head).  With a = 8, b = 0.75, c = 4 the mean SINK mass is about
  30x the content roles' and KEY tokens carry about 1.3x the VALUE mass
  (the per-role mass ratios of Section 3, 'Mass concentration').
"""

from __future__ import annotations

import dataclasses
from typing import Optional

import numpy as np
import torch

ROLE_SINK, ROLE_KEY, ROLE_VALUE, ROLE_OTHER = 0, 1, 2, 3
ROLE_NAMES = ("SINK", "KEY", "VALUE", "OTHER")
N_ROLES = 4

# Content-role weights of the combined method (Section 4.1): VALUE 0.70,
# DELIM 0.20 and WS 0.05 (merged into SINK), PROSE 0.05 (OTHER); KEY is the
# tuned alpha_KEY, passed separately.
PAPER_ALPHA = (0.25, 0.0, 0.70, 0.05)
ALPHA_KEY_SAFE = 0.02   # the cross-model safe default (Section 5)

# The paper's six-label taxonomy (Section 3) with its policy (Section 4.1);
# HEADER, a schema label like KEY, takes alpha_KEY as well.
SIX_ROLE_NAMES = ("KEY", "VALUE", "DELIM", "HEADER", "PROSE", "WS")


def paper_alpha6(alpha_key: float) -> tuple:
    return (alpha_key, 0.70, 0.20, alpha_key, 0.05, 0.05)

SINK_SHIFT = 8.0    # a
KEY_SHIFT = 0.75    # b
QUERY_SHIFT = 4.0   # c


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    kind: str                 # "snapkv" or "h2o"
    L: int
    b: int
    Hq: int
    Hkv: int
    d: int
    n: int                    # tokens per sequence (dense) or the largest (varlen)
    W: int
    pool_k: int
    budgets: tuple
    max_depth: int
    key_run: tuple
    value_run: tuple
    seqlens: Optional[tuple] = None

    @property
    def G(self) -> int:
        return self.Hq // self.Hkv

    @property
    def varlen(self) -> bool:
        return self.seqlens is not None

    @property
    def n_units(self) -> int:
        return self.L * self.b * self.Hkv

    def lengths(self):
        return list(self.seqlens) if self.varlen else [self.n] * self.b

    def scaled(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


def ragged_seqlens(count: int = 64, lo: int = 1024, hi: int = 16384, seed: int = 0) -> tuple:
    rng = np.random.default_rng(np.random.SeedSequence([seed, 0x5EED]))
    return tuple(int(x) for x in rng.integers(lo, hi + 1, size=count))


WORKLOADS = {
    "tiny": Workload("tiny", "snapkv", 1, 1, 8, 2, 64, 2048, 32, 7, (0.05,), 4, (3, 5), (1, 3)),
    "llama8b": Workload("llama8b", "snapkv", 32, 1, 32, 8, 128, 8192, 32, 7,
                        (0.05, 0.10, 0.20, 0.30, 0.50), 4, (3, 5), (1, 3)),
    "long": Workload("long", "snapkv", 32, 4, 32, 8, 128, 32768, 64, 7, (0.10,), 8, (2, 3), (2, 4)),
    "h2o": Workload("h2o", "h2o", 32, 2, 32, 8, 128, 8192, 0, 1, (0.05,), 4, (3, 5), (1, 3)),
    "ragged": Workload("ragged", "snapkv", 28, 64, 28, 4, 128, 16384, 32, 7, (0.10,), 4, (3, 5), (1, 3),
                       seqlens=ragged_seqlens()),
}


# ---------------------------------------------------------------------------
# role streams
# ---------------------------------------------------------------------------

def json_roles(n: int, seed: int, max_depth: int = 4, key_run=(3, 5), value_run=(1, 3),
               tail: int = 48, prefix: int = 32) -> np.ndarray:
    """Role label per token of one synthetic prompt (uint8, length n)."""
    rng = np.random.default_rng(np.random.SeedSequence([seed, n, max_depth, 0x4A53]))
    out: list[int] = []
    body = max(0, n - tail)
    out.extend([ROLE_OTHER] * min(prefix, body))

    def emit_object(depth: int):
        out.append(ROLE_SINK)                                   # '{'
        for _ in range(int(rng.integers(2, 7))):
            if len(out) >= body:
                return
            out.append(ROLE_SINK)                               # newline + indent
            out.extend([ROLE_KEY] * int(rng.integers(key_run[0], key_run[1] + 1)))
            out.append(ROLE_SINK)                               # ':'
            if depth < max_depth and rng.random() < 0.4:
                emit_object(depth + 1)
            else:
                out.extend([ROLE_VALUE] * int(rng.integers(value_run[0], value_run[1] + 1)))
            out.append(ROLE_SINK)                               # ','
        out.append(ROLE_SINK)                                   # newline
        out.append(ROLE_SINK)                                   # '}'

    while len(out) < body:
        emit_object(1)
    roles = out[:body] + [ROLE_OTHER] * (n - body)
    return np.asarray(roles[:n], dtype=np.uint8)


def workload_roles(w: Workload, seed: int = 0) -> np.ndarray:
    """Dense [b][n] or packed [T] roles for a workload."""
    seqs = [json_roles(n, seed * 1000003 + s, w.max_depth, w.key_run, w.value_run,
                       tail=max(w.W, 48)) for s, n in enumerate(w.lengths())]
    if w.varlen:
        return np.concatenate(seqs) if seqs else np.zeros(0, np.uint8)
    return np.stack(seqs)


# ---------------------------------------------------------------------------
# Q / K / V
# ---------------------------------------------------------------------------

def _gen(device, seed: int, stream: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed((seed * 0x9E3779B1 + stream * 0x85EBCA77) & 0x7FFFFFFFFFFFFFFF)
    return g


def _directions(w: Workload, seed: int, device) -> torch.Tensor:
    u = torch.randn(w.L, w.Hkv, w.d, generator=_gen(device, seed, 7), device=device)
    return u / u.norm(dim=-1, keepdim=True)


def _role_shift(roles: torch.Tensor) -> torch.Tensor:
    shift = torch.zeros(roles.shape, dtype=torch.float32, device=roles.device)
    shift[roles == ROLE_SINK] = SINK_SHIFT
    shift[roles == ROLE_KEY] = KEY_SHIFT
    return shift


def make_kv(w: Workload, roles: np.ndarray, seed: int = 0, device="cpu", with_v: bool = True):
    """K (and V) as bf16 tensors: dense [L][b][Hkv][n][d] or packed
    [L][T][Hkv][d].  Generated one layer at a time to bound temporaries."""
    u = _directions(w, seed, device)
    r = torch.as_tensor(roles.astype(np.int64), device=device)
    shift = _role_shift(r)
    gk, gv = _gen(device, seed, 1), _gen(device, seed, 2)
    if w.varlen:
        T = r.shape[0]
        K = torch.empty(w.L, T, w.Hkv, w.d, dtype=torch.bfloat16, device=device)
        V = torch.empty_like(K) if with_v else None
        for l in range(w.L):
            z = torch.randn(T, w.Hkv, w.d, generator=gk, device=device)
            z += shift[:, None, None] * u[l][None, :, :]
            K[l] = z.to(torch.bfloat16)
            if with_v:
                V[l] = torch.randn(T, w.Hkv, w.d, generator=gv, device=device).to(torch.bfloat16)
    else:
        K = torch.empty(w.L, w.b, w.Hkv, w.n, w.d, dtype=torch.bfloat16, device=device)
        V = torch.empty_like(K) if with_v else None
        for l in range(w.L):
            z = torch.randn(w.b, w.Hkv, w.n, w.d, generator=gk, device=device)
            z += shift[:, None, :, None] * u[l][None, :, None, :]
            K[l] = z.to(torch.bfloat16)
            if with_v:
                V[l] = torch.randn(w.b, w.Hkv, w.n, w.d, generator=gv, device=device).to(torch.bfloat16)
    return K, V


def make_q_window(w: Workload, seed: int = 0, device="cpu") -> torch.Tensor:
    """SnapKV window queries [L][b][Hq][W][d] (bf16): z + c u of the head's KV
    direction."""
    u = _directions(w, seed, device)
    z = torch.randn(w.L, w.b, w.Hq, w.W, w.d, generator=_gen(device, seed, 3), device=device)
    uq = u.repeat_interleave(w.G, dim=1)                      # [L][Hq][d]
    z += QUERY_SHIFT * uq[:, None, :, None, :]
    return z.to(torch.bfloat16)


def make_q_decode(w: Workload, seed: int = 0, device="cpu") -> torch.Tensor:
    """One decode query per sequence and head [L][b][Hq][d] (bf16), drawn like
    the window queries."""
    u = _directions(w, seed, device)
    z = torch.randn(w.L, w.b, w.Hq, w.d, generator=_gen(device, seed, 5), device=device)
    z += QUERY_SHIFT * u.repeat_interleave(w.G, dim=1)[:, None, :, :]
    return z.to(torch.bfloat16)


def make_q_full(w: Workload, seed: int = 0, device="cpu") -> torch.Tensor:
    """All prefill queries (H2O): dense [L][b][Hq][n][d] or packed [L][T][Hq][d]."""
    u = _directions(w, seed, device)
    uq = u.repeat_interleave(w.G, dim=1)
    g = _gen(device, seed, 4)
    if w.varlen:
        T = sum(w.lengths())
        Q = torch.empty(w.L, T, w.Hq, w.d, dtype=torch.bfloat16, device=device)
        for l in range(w.L):
            z = torch.randn(T, w.Hq, w.d, generator=g, device=device)
            z += QUERY_SHIFT * uq[l][None, :, :]
            Q[l] = z.to(torch.bfloat16)
    else:
        Q = torch.empty(w.L, w.b, w.Hq, w.n, w.d, dtype=torch.bfloat16, device=device)
        for l in range(w.L):
            z = torch.randn(w.b, w.Hq, w.n, w.d, generator=g, device=device)
            z += QUERY_SHIFT * uq[l][None, :, None, :]
            Q[l] = z.to(torch.bfloat16)
    return Q


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """Host copy of a bf16 tensor as uint16 bit patterns."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
