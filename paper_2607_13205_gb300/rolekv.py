"""Python binding of librolekv: argument marshalling only.

Every function here forwards torch tensors' device pointers and the current
CUDA stream to the C ABI of the same name (include/rolekv.h); all work runs
in the library's sm_103a kernels.  There is no fallback: if the shared
library is missing the first call raises.
"""

from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import torch

# ROLEKV_CHECKED=1 in the environment selects the checked build (every
# computed global access checked against its buffer's extent; a miss sets
# STATUS_BOUNDS and is skipped), which has the same entry points.
_LIB_NAME = "librolekv_checked.so" if os.environ.get("ROLEKV_CHECKED") == "1" else "librolekv.so"
_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), _LIB_NAME)

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_WORKSPACE, ERR_CUDA = 0, 1, 2, 3, 4
STATUS_NONFINITE, STATUS_BAD_INDEX, STATUS_TIMEOUT, STATUS_BOUNDS = 1, 2, 4, 8
POLICY_ROLE_QUOTA, POLICY_GLOBAL, POLICY_FAIR, POLICY_SLACK, POLICY_CEIL = 0, 1, 2, 3, 4
MAX_ROLES = 8
SELECT_MAX_N = 262144
OP_SNAPKV, OP_H2O, OP_COMPRESS = 0, 1, 2


class RolekvError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"rolekv error {code}: {msg}")
        self.code = code


class Tensor(ctypes.Structure):
    _fields_ = [("ptr", ctypes.c_void_p), ("s_layer", ctypes.c_int64), ("s_seq", ctypes.c_int64),
                ("s_head", ctypes.c_int64), ("s_tok", ctypes.c_int64)]


class BatchDesc(ctypes.Structure):
    _fields_ = [("L", ctypes.c_int32), ("b", ctypes.c_int32), ("Hq", ctypes.c_int32),
                ("Hkv", ctypes.c_int32), ("d", ctypes.c_int32), ("n_max", ctypes.c_int32),
                ("seqlens_host", ctypes.POINTER(ctypes.c_int32)),
                ("cu_seqlens_dev", ctypes.c_void_p), ("kept_extra", ctypes.c_int32)]


class SelectParams(ctypes.Structure):
    _fields_ = [("n_roles", ctypes.c_int32), ("alpha", ctypes.c_float * MAX_ROLES),
                ("key_role", ctypes.c_int32), ("alpha_key", ctypes.c_float),
                ("budget", ctypes.c_float), ("policy", ctypes.c_int32),
                ("ban_mask", ctypes.c_uint32), ("keep_last", ctypes.c_int32)]


_lib = None

# (name, restype, argtypes) of every exported function
_SIGNATURES = [
    ("rolekv_kept_count", ctypes.c_int64, [ctypes.c_int64, ctypes.c_float]),
    ("rolekv_kept_rows", ctypes.c_int64, [ctypes.c_int64, ctypes.c_float, ctypes.c_int32]),
    ("rolekv_workspace_size", ctypes.c_int,
     [ctypes.c_int, ctypes.POINTER(BatchDesc), ctypes.c_int32, ctypes.POINTER(ctypes.c_size_t)]),
    ("snapkv_score", ctypes.c_int,
     [ctypes.POINTER(BatchDesc), Tensor, Tensor, ctypes.c_int32, ctypes.c_int32, ctypes.c_float,
      ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t,
      ctypes.c_void_p, ctypes.c_void_p]),
    ("snapkv_score_noalloc", ctypes.c_int,
     [ctypes.POINTER(BatchDesc), Tensor, Tensor, ctypes.c_int32, ctypes.c_int32, ctypes.c_float,
      ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]),
    ("quest_score", ctypes.c_int,
     [ctypes.POINTER(BatchDesc), Tensor, Tensor, ctypes.c_int32, ctypes.c_int32, ctypes.c_void_p,
      ctypes.c_void_p]),
    ("rolekv_selftest_wait", ctypes.c_int, [ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p]),
    ("rolekv_decode_workspace_size", ctypes.c_int,
     [ctypes.POINTER(BatchDesc), ctypes.c_float, ctypes.POINTER(ctypes.c_size_t)]),
    ("decode_attention", ctypes.c_int,
     [ctypes.POINTER(BatchDesc), Tensor, Tensor, Tensor, ctypes.c_void_p, ctypes.c_float,
      ctypes.c_float, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p,
      ctypes.c_void_p]),
    ("h2o_score", ctypes.c_int,
     [ctypes.POINTER(BatchDesc), Tensor, Tensor, ctypes.c_float, ctypes.c_void_p, ctypes.c_void_p,
      ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p, ctypes.c_void_p]),
    ("rolekv_selftest_score_timeout", ctypes.c_int, [ctypes.c_int64]),
    ("rolekv_checked_build", ctypes.c_int, []),
    ("rolekv_selftest_shrink_extent", ctypes.c_int, [ctypes.c_int64]),
    ("role_alloc_select", ctypes.c_int,
     [ctypes.POINTER(BatchDesc), ctypes.c_void_p, ctypes.c_void_p, ctypes.POINTER(SelectParams),
      ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
      ctypes.c_void_p]),
    ("kv_compact", ctypes.c_int,
     [ctypes.POINTER(BatchDesc), Tensor, Tensor, ctypes.c_void_p, ctypes.c_float, ctypes.c_void_p,
      ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]),
    ("rolekv_compress", ctypes.c_int,
     [ctypes.POINTER(BatchDesc), Tensor, Tensor, Tensor, ctypes.c_int32, ctypes.c_int32,
      ctypes.c_float, ctypes.c_void_p, ctypes.c_void_p, ctypes.POINTER(SelectParams),
      ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
      ctypes.c_size_t, ctypes.c_void_p, ctypes.c_void_p]),
    ("rolekv_set_stage_events", ctypes.c_int, [ctypes.POINTER(ctypes.c_void_p), ctypes.c_int32]),
    ("rolekv_last_error", ctypes.c_char_p, []),
    ("rolekv_version", ctypes.c_char_p, []),
]


def library_path() -> str:
    return _LIB_PATH


def lib():
    """The loaded librolekv (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"{_LIB_PATH} is missing: build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        L = ctypes.CDLL(_LIB_PATH)
        for name, res, args in _SIGNATURES:
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def _check(rc: int):
    if rc != OK:
        raise RolekvError(rc, lib().rolekv_last_error().decode())


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


# ---------------------------------------------------------------- descriptors

class Batch:
    """Shapes of one call.  seqlens (list of ints) makes it a varlen batch; the
    device copy of the prefix sums is created here, once.  kept_extra widens
    every kept row beyond ceil(B n) (the ceiling policy needs it)."""

    def __init__(self, L, b, Hq, Hkv, d, n_max, seqlens: Optional[Sequence[int]] = None,
                 device="cuda", kept_extra: int = 0):
        self.L, self.b, self.Hq, self.Hkv, self.d, self.n_max = L, b, Hq, Hkv, d, n_max
        self.kept_extra = int(kept_extra)
        self.seqlens = list(seqlens) if seqlens is not None else None
        self._host = None
        self.cu_seqlens = None
        if self.seqlens is not None:
            self._host = (ctypes.c_int32 * len(self.seqlens))(*self.seqlens)
            cu = [0]
            for n in self.seqlens:
                cu.append(cu[-1] + n)
            self.cu_seqlens = torch.tensor(cu, dtype=torch.int32, device=device)
        self.desc = BatchDesc(L, b, Hq, Hkv, d, n_max,
                              self._host if self._host is not None else None,
                              ctypes.c_void_p(self.cu_seqlens.data_ptr()) if self.cu_seqlens is not None else None,
                              self.kept_extra)

    @property
    def varlen(self) -> bool:
        return self.seqlens is not None

    @property
    def T(self) -> int:
        return sum(self.seqlens) if self.varlen else self.b * self.n_max

    @property
    def n_units(self) -> int:
        return self.L * self.b * self.Hkv

    def score_shape(self):
        return (self.L, self.Hkv, self.T) if self.varlen else (self.L, self.b, self.Hkv, self.n_max)

    def role_shape(self):
        return (self.T,) if self.varlen else (self.b, self.n_max)

    def kept_shape(self, budget: float):
        if self.varlen:
            return (self.L, self.Hkv, sum(kept_rows(n, budget, self.kept_extra) for n in self.seqlens))
        return (self.L, self.b, self.Hkv, kept_rows(self.n_max, budget, self.kept_extra))


def tensor_desc(t: torch.Tensor, packed: bool = False) -> Tensor:
    """Strides of a 5-D [L][b][H][n][d] tensor, or of a packed 4-D [L][T][H][d]
    tensor, as a rolekv_tensor."""
    if t.dtype != torch.bfloat16:
        raise TypeError("rolekv tensors are bf16")
    if t.stride(-1) != 1:
        raise ValueError("the head-dim axis must be contiguous")
    if packed:
        if t.dim() != 4:
            raise ValueError("packed tensors are [L][T][H][d]")
        sl, st, sh, _ = t.stride()
        return Tensor(t.data_ptr(), sl, 0, sh, st)
    if t.dim() != 5:
        raise ValueError("dense tensors are [L][b][H][n][d]")
    sl, ss, sh, st, _ = t.stride()
    return Tensor(t.data_ptr(), sl, ss, sh, st)


def select_params(budget: float, alpha: Sequence[float], alpha_key: float = 0.0, key_role: int = 1,
                  policy: int = POLICY_ROLE_QUOTA, ban_mask: int = 0,
                  keep_last: int = 0) -> SelectParams:
    al = (ctypes.c_float * MAX_ROLES)(*([float(x) for x in alpha] + [0.0] * (MAX_ROLES - len(alpha))))
    return SelectParams(len(alpha), al, key_role, alpha_key, budget, policy, ban_mask, keep_last)


# ----------------------------------------------------------------- entry points

def kept_count(n: int, budget: float) -> int:
    return int(lib().rolekv_kept_count(int(n), float(budget)))


def kept_rows(n: int, budget: float, kept_extra: int = 0) -> int:
    return int(lib().rolekv_kept_rows(int(n), float(budget), int(kept_extra)))


def workspace_size(op: int, batch: Batch, W: int = 0) -> int:
    out = ctypes.c_size_t(0)
    _check(lib().rolekv_workspace_size(op, ctypes.byref(batch.desc), W, ctypes.byref(out)))
    return int(out.value)


def workspace(op: int, batch: Batch, W: int = 0, device="cuda") -> torch.Tensor:
    return torch.empty(max(workspace_size(op, batch, W), 256), dtype=torch.uint8, device=device)


def snapkv_score(batch: Batch, q_win: torch.Tensor, k: torch.Tensor, W: int, pool_k: int,
                 scores: torch.Tensor, scores_prepool: Optional[torch.Tensor] = None,
                 lse_win: Optional[torch.Tensor] = None, scale: float = 0.0,
                 ws: Optional[torch.Tensor] = None, status: Optional[torch.Tensor] = None,
                 stream=None) -> torch.Tensor:
    if ws is None:
        ws = workspace(OP_SNAPKV, batch, W, device=k.device)
    _check(lib().snapkv_score(ctypes.byref(batch.desc), tensor_desc(q_win), tensor_desc(k, batch.varlen),
                              W, pool_k, scale, _ptr(lse_win), _ptr(scores), _ptr(scores_prepool),
                              _ptr(ws), ws.numel(), _ptr(status), _stream(stream)))
    return scores


def snapkv_score_noalloc(batch: Batch, q_win: torch.Tensor, k: torch.Tensor, W: int, pool_k: int,
                         scores: torch.Tensor, scores_prepool: Optional[torch.Tensor] = None,
                         lse_win: Optional[torch.Tensor] = None, scale: float = 0.0,
                         status: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """snapkv_score for callers that cannot allocate device memory: no
    workspace argument, the library's own static scratch is used instead
    (see rolekv.h for its limit and sharing rules)."""
    _check(lib().snapkv_score_noalloc(ctypes.byref(batch.desc), tensor_desc(q_win),
                                      tensor_desc(k, batch.varlen), W, pool_k, scale, _ptr(lse_win),
                                      _ptr(scores), _ptr(scores_prepool), _ptr(status), _stream(stream)))
    return scores


def quest_score(batch: Batch, q_win: torch.Tensor, k: torch.Tensor, W: int, page: int,
                scores: torch.Tensor, stream=None) -> torch.Tensor:
    _check(lib().quest_score(ctypes.byref(batch.desc), tensor_desc(q_win, False),
                             tensor_desc(k, batch.varlen), W, page, _ptr(scores), _stream(stream)))
    return scores


def selftest_wait(limit_ns: int, status: torch.Tensor, stream=None) -> None:
    _check(lib().rolekv_selftest_wait(int(limit_ns), _ptr(status), _stream(stream)))


def decode_workspace(batch: Batch, budget: float, device="cuda") -> torch.Tensor:
    out = ctypes.c_size_t(0)
    _check(lib().rolekv_decode_workspace_size(ctypes.byref(batch.desc), budget, ctypes.byref(out)))
    return torch.empty(max(int(out.value), 256), dtype=torch.uint8, device=device)


def cache_desc(t: torch.Tensor, batch: Batch, compacted: bool) -> Tensor:
    """Strides of a cache tensor: kv_compact's output (compacted=True:
    dense [L][b][Hkv][K][d], varlen [L][Hkv][Ktot][d]) or an uncompacted K/V
    in the library's own layouts."""
    if compacted and batch.varlen:
        return tensor_desc(t.transpose(1, 2), True)
    return tensor_desc(t, batch.varlen)


def decode_attention(batch: Batch, q: torch.Tensor, k_cache: torch.Tensor, v_cache: torch.Tensor,
                     keep_idx: Optional[torch.Tensor], budget: float, out: torch.Tensor,
                     compacted: bool = True, scale: float = 0.0, ws: Optional[torch.Tensor] = None,
                     status: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """q bf16 [L][b][Hq][d] -> out fp32 [L][b][Hq][d]."""
    if ws is None:
        ws = decode_workspace(batch, budget, device=q.device)
    if q.dtype != torch.bfloat16 or q.dim() != 4 or q.stride(-1) != 1:
        raise ValueError("q is a bf16 [L][b][Hq][d] tensor with a contiguous last axis")
    sl, ss, sh, _ = q.stride()
    qd = Tensor(q.data_ptr(), sl, ss, sh, q.shape[-1])
    _check(lib().decode_attention(ctypes.byref(batch.desc), qd, cache_desc(k_cache, batch, compacted),
                                  cache_desc(v_cache, batch, compacted), _ptr(keep_idx), budget, scale,
                                  _ptr(out), _ptr(ws), ws.numel(), _ptr(status), _stream(stream)))
    return out


def h2o_score(batch: Batch, q: torch.Tensor, k: torch.Tensor, scores: torch.Tensor, scale: float = 0.0,
              lse: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None,
              status: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """lse: optional fp32 natural-log normalisers of every query row (dense
    [L][b][Hq][n], varlen [L][Hq][T]); given, the score is one pass over K."""
    if ws is None:
        ws = workspace(OP_H2O, batch, 0, device=k.device)
    _check(lib().h2o_score(ctypes.byref(batch.desc), tensor_desc(q, batch.varlen),
                           tensor_desc(k, batch.varlen), scale, _ptr(lse), _ptr(scores), _ptr(ws),
                           ws.numel(), _ptr(status), _stream(stream)))
    return scores


def selftest_score_timeout(limit_ns: int) -> None:
    """Arm the next two-pass SnapKV score on this thread to time out at its
    per-unit meeting point after limit_ns (diagnostic; see rolekv.h)."""
    _check(lib().rolekv_selftest_score_timeout(int(limit_ns)))


def checked_build() -> bool:
    """Whether the loaded library is the checked build."""
    return lib().rolekv_checked_build() == 1


def selftest_shrink_extent(rows: int) -> None:
    """Checked build only: the next kv_compact on this thread takes its output
    extent as `rows` rows smaller, so its checks on the last rows fire
    (diagnostic; see rolekv.h)."""
    _check(lib().rolekv_selftest_shrink_extent(int(rows)))


def role_alloc_select(batch: Batch, scores: torch.Tensor, roles: torch.Tensor, params: SelectParams,
                      keep_idx: torch.Tensor, pool_k: int = 1, keep_mask: Optional[torch.Tensor] = None,
                      kept_per_role: Optional[torch.Tensor] = None, status: Optional[torch.Tensor] = None,
                      stream=None) -> torch.Tensor:
    _check(lib().role_alloc_select(ctypes.byref(batch.desc), _ptr(scores), _ptr(roles), ctypes.byref(params),
                                   pool_k, _ptr(keep_idx), _ptr(keep_mask), _ptr(kept_per_role),
                                   _ptr(status), _stream(stream)))
    return keep_idx


def kv_compact(batch: Batch, k: torch.Tensor, v: torch.Tensor, keep_idx: torch.Tensor, budget: float,
               k_out: torch.Tensor, v_out: torch.Tensor, status: Optional[torch.Tensor] = None,
               stream=None):
    _check(lib().kv_compact(ctypes.byref(batch.desc), tensor_desc(k, batch.varlen),
                            tensor_desc(v, batch.varlen), _ptr(keep_idx), budget, _ptr(k_out),
                            _ptr(v_out), _ptr(status), _stream(stream)))
    return k_out, v_out


def rolekv_compress(batch: Batch, q_win: torch.Tensor, k: torch.Tensor, v: torch.Tensor, W: int,
                    pool_k: int, roles: torch.Tensor, params: SelectParams, keep_idx: torch.Tensor,
                    k_out: torch.Tensor, v_out: torch.Tensor, ws: torch.Tensor,
                    kept_per_role: Optional[torch.Tensor] = None, lse_win: Optional[torch.Tensor] = None,
                    scale: float = 0.0, status: Optional[torch.Tensor] = None, stream=None):
    _check(lib().rolekv_compress(ctypes.byref(batch.desc), tensor_desc(q_win), tensor_desc(k, batch.varlen),
                                 tensor_desc(v, batch.varlen), W, pool_k, scale, _ptr(lse_win), _ptr(roles),
                                 ctypes.byref(params), _ptr(keep_idx), _ptr(k_out), _ptr(v_out),
                                 _ptr(kept_per_role), _ptr(ws), ws.numel(), _ptr(status), _stream(stream)))
    return keep_idx, k_out, v_out


def set_stage_events(events: Sequence[torch.cuda.Event]):
    """Record events[i] after the i-th kernel launch of every later call on
    this thread (empty sequence: off).  The events must have been recorded
    once so that they exist."""
    arr = (ctypes.c_void_p * max(1, len(events)))(*[ctypes.c_void_p(e.cuda_event) for e in events])
    _check(lib().rolekv_set_stage_events(arr, len(events)))


def compact_shape(batch: Batch, budget: float):
    return batch.kept_shape(budget) + (batch.d,)
