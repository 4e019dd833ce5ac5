"""The C ABI on the CPU: the library loads, exports every function that
include/rolekv.h declares, and rejects bad arguments on the host before
touching the GPU."""

import ctypes
import os
import re

import numpy as np
import pytest

from oracle import rolekv_oracle as O
from paper_2607_13205_gb300 import build as B
from paper_2607_13205_gb300 import rolekv as R

HEADER = os.path.join(B.ROOT, "include", "rolekv.h")


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(B.LIB_PATH):
        B.build()
    return R.lib()


def _declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\*?\s*([A-Za-z_][A-Za-z0-9_]*)\s*\(",
                       text, flags=re.M)
    return sorted(set(n for n in names if n not in ("if", "while", "for", "sizeof")))


def test_header_declares_the_four_calls():
    names = _declared_functions()
    for n in ("snapkv_score", "h2o_score", "role_alloc_select", "kv_compact"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    names = _declared_functions()
    assert len(names) >= 8
    for n in names:
        assert hasattr(lib, n), f"{n} declared in rolekv.h but not exported"


def test_checked_build_loads_and_exports_every_symbol(lib):
    """The checked library (-DROLEKV_CHECKED) is built beside the plain one,
    exports the same entry points and says which it is; its extent self-test
    is refused by the plain build.  Host calls only."""
    if not os.path.exists(B.CHECKED_LIB_PATH):
        B.build(checked=True)
    chk = ctypes.CDLL(B.CHECKED_LIB_PATH)
    for n in _declared_functions():
        assert hasattr(chk, n), f"{n} declared in rolekv.h but not exported by the checked build"
    assert chk.rolekv_checked_build() == 1
    assert lib.rolekv_checked_build() == 0
    shrink = chk.rolekv_selftest_shrink_extent
    shrink.argtypes = [ctypes.c_int64]
    assert shrink(0) == R.ERR_INVALID_ARG          # (an out-of-range count arms nothing)
    assert lib.rolekv_selftest_shrink_extent(1) == R.ERR_UNSUPPORTED


def test_kept_count_matches_oracle(lib):
    for n in (0, 1, 7, 100, 2048, 8192, 32768, 40960, 123457):
        for b in (0.05, 0.1, 0.2, 0.3, 0.5, 0.75, 1.0, 0.333):
            assert R.kept_count(n, b) == O.kept_count(n, b), (n, b)
    assert R.kept_count(10, 0.0) == -1
    assert R.kept_count(10, 1.5) == -1
    assert R.kept_count(-1, 0.5) == -1


def test_kept_rows_matches_oracle(lib):
    for extra in (0, 1, 3, 7, 100000):
        ob = O.Batch(1, 1, 1, 1, 8, 1, kept_extra=extra)
        for n in (0, 1, 7, 100, 2048, 32768, 123457):
            for b in (0.05, 0.1, 0.333, 1.0):
                assert R.kept_rows(n, b, extra) == ob.kept_rows(n, b), (n, b, extra)
    assert R.kept_rows(10, 0.5, -1) == -1
    assert R.kept_rows(10, 0.0, 2) == -1


def _batch(**kw):
    d = dict(L=2, b=3, Hq=8, Hkv=2, d=128, n_max=1000)
    d.update(kw)
    return R.BatchDesc(d["L"], d["b"], d["Hq"], d["Hkv"], d["d"], d["n_max"], None, None)


def _ws(op, batch, W):
    out = ctypes.c_size_t(0)
    rc = R.lib().rolekv_workspace_size(op, ctypes.byref(batch), W, ctypes.byref(out))
    return rc, out.value


def test_workspace_size(lib):
    rc, sz = _ws(0, _batch(), 32)
    assert rc == 0 and sz >= 2 * 3 * 2 * 1000 * 4
    rc, sz_h2o = _ws(1, _batch(), 0)
    assert rc == 0 and sz_h2o > 0
    assert _ws(0, _batch(), 12)[0] == R.ERR_UNSUPPORTED        # W not a multiple of 8
    assert _ws(0, _batch(Hq=16, Hkv=2), 64)[0] == R.ERR_UNSUPPORTED   # W*G > 256
    assert _ws(0, _batch(d=96), 32)[0] == R.ERR_UNSUPPORTED
    assert _ws(0, _batch(Hq=7, Hkv=2), 32)[0] == R.ERR_INVALID_ARG
    assert _ws(1, _batch(Hq=18, Hkv=2), 0)[0] == R.ERR_UNSUPPORTED   # H2O G > 8
    assert _ws(9, _batch(), 32)[0] == R.ERR_INVALID_ARG


def test_host_rejects_bad_arguments(lib):
    b = _batch()
    t = R.Tensor(16, 0, 0, 0, 128)        # fake, never dereferenced: checks fail first
    f = ctypes.c_void_p(256)
    rc = lib.snapkv_score(ctypes.byref(b), t, t, 32, 4, 0.0, None, f, None, f, 1 << 30, None, None)
    assert rc == R.ERR_UNSUPPORTED                                      # even pool width
    rc = lib.snapkv_score(ctypes.byref(b), t, t, 32, 7, 0.0, None, None, None, f, 1 << 30, None, None)
    assert rc == R.ERR_INVALID_ARG                                      # no output
    bad = R.Tensor(24, 0, 0, 0, 128)       # misaligned pointer
    rc = lib.snapkv_score(ctypes.byref(b), bad, t, 32, 7, 0.0, None, f, None, f, 1 << 30, None, None)
    assert rc == R.ERR_INVALID_ARG
    assert b"aligned" in lib.rolekv_last_error()
    p = R.select_params(0.1, [0.25, 0.0, 0.7, 0.05])
    rc = lib.role_alloc_select(ctypes.byref(b), f, f, ctypes.byref(p), 2, f, None, None, None, None)
    assert rc == R.ERR_UNSUPPORTED                                      # even pool width
    p_bad = R.select_params(1.5, [0.25, 0.0, 0.7, 0.05])
    rc = lib.role_alloc_select(ctypes.byref(b), f, f, ctypes.byref(p_bad), 1, f, None, None, None, None)
    assert rc == R.ERR_INVALID_ARG
    p_neg = R.select_params(0.1, [0.25, 0.0, -0.7, 0.05])
    rc = lib.role_alloc_select(ctypes.byref(b), f, f, ctypes.byref(p_neg), 1, f, None, None, None, None)
    assert rc == R.ERR_INVALID_ARG
    p_pol = R.select_params(0.1, [0.25, 0.0, 0.7, 0.05], policy=5)
    rc = lib.role_alloc_select(ctypes.byref(b), f, f, ctypes.byref(p_pol), 1, f, None, None, None, None)
    assert rc == R.ERR_INVALID_ARG                                      # unknown policy
    # the ceiling policy over 3 weighted roles needs rows 2 slots wider
    p_ceil = R.select_params(0.1, [0.25, 0.0, 0.7, 0.05], policy=R.POLICY_CEIL)
    narrow = _batch()
    narrow.kept_extra = 1
    rc = lib.role_alloc_select(ctypes.byref(narrow), f, f, ctypes.byref(p_ceil), 1, f, None, None, None, None)
    assert rc == R.ERR_INVALID_ARG and b"kept_extra >= 2" in lib.rolekv_last_error()
    # the one-call path applies the same check before it launches anything
    rc = lib.rolekv_compress(ctypes.byref(narrow), R.Tensor(256, 0, 32 * 128, 8 * 128, 128),
                             R.Tensor(256, 2 * 1000 * 128, 1000 * 128, 0, 128), t, 32, 7, 0.0, None, f,
                             ctypes.byref(p_ceil), f, f, f, None, f, 1 << 30, None, None)
    assert rc == R.ERR_INVALID_ARG and b"kept_extra" in lib.rolekv_last_error()
    neg = _batch()
    neg.kept_extra = -1
    rc = lib.kv_compact(ctypes.byref(neg), t, t, f, 0.1, f, f, None, None)
    assert rc == R.ERR_INVALID_ARG and b"kept_extra" in lib.rolekv_last_error()
    p_floor = R.select_params(0.1, [0.25, 0.0, 0.7, 0.05], keep_last=-1)
    rc = lib.role_alloc_select(ctypes.byref(b), f, f, ctypes.byref(p_floor), 1, f, None, None, None, None)
    assert rc == R.ERR_INVALID_ARG                                      # negative floor
    assert b"keep_last" in lib.rolekv_last_error()
    big = _batch(n_max=R.SELECT_MAX_N + 1)
    rc = lib.role_alloc_select(ctypes.byref(big), f, f, ctypes.byref(p), 1, f, None, None, None, None)
    assert rc == R.ERR_UNSUPPORTED
    rc = lib.kv_compact(ctypes.byref(_batch(d=96)), t, t, f, 0.1, f, f, None, None)
    assert rc == R.ERR_UNSUPPORTED
    rc = lib.kv_compact(ctypes.byref(b), t, t, f, 0.1, None, f, None, None)
    assert rc == R.ERR_INVALID_ARG
    lens = (ctypes.c_int32 * 3)(10, 2000, 5)
    vb = R.BatchDesc(2, 3, 8, 2, 128, 1000, lens, ctypes.c_void_p(64))
    rc = lib.kv_compact(ctypes.byref(vb), t, t, f, 0.1, f, f, None, None)
    assert rc == R.ERR_INVALID_ARG                                      # length > n_max
    assert b"seqlens" in lib.rolekv_last_error()


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(R, "_LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(R, "_lib", None)
    with pytest.raises(RuntimeError, match="missing"):
        R.kept_count(10, 0.5)

def test_struct_layouts_match_the_header(tmp_path):
    """The binding's ctypes structs have the sizes and field offsets that a C
    compiler gives the header's structs (the header also compiles as C99)."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    fields = {"rolekv_batch": [f for f, _ in R.BatchDesc._fields_],
              "rolekv_select_params": [f for f, _ in R.SelectParams._fields_],
              "rolekv_tensor": [f for f, _ in R.Tensor._fields_]}
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "rolekv.h"', "int main(void) {"]
    for st, fs in fields.items():
        lines.append(f'  printf("{st} size %zu\\n", sizeof({st}));')
        for f in fs:
            lines.append(f'  printf("{st} {f} %zu\\n", offsetof({st}, {f}));')
    lines += ["  return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    subprocess.run([cc, "-std=c99", "-Wall", "-Werror", "-I", inc, str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split("\n")
    got = {tuple(l.split()[:-1]): int(l.split()[-1]) for l in out if l}
    for st, cls in (("rolekv_batch", R.BatchDesc), ("rolekv_select_params", R.SelectParams),
                    ("rolekv_tensor", R.Tensor)):
        assert got[(st, "size")] == ctypes.sizeof(cls), st
        for f in fields[st]:
            assert got[(st, f)] == getattr(cls, f).offset, (st, f)


_NOALLOC_REJECTS = r'''
import ctypes, sys
sys.path.insert(0, sys.argv[1])
from paper_2607_13205_gb300 import rolekv as R
lib = R.lib()
t = R.Tensor(16, 0, 0, 0, 128)          # fake, never dereferenced: checks fail first
f = ctypes.c_void_p(256)
# 64 layers x 64 sequences x 8 KV heads at 16384 tokens need more scratch
# than the static array holds
b = R.BatchDesc(64, 64, 32, 8, 128, 16384, None, None)
rc = lib.snapkv_score_noalloc(ctypes.byref(b), t, t, 32, 1, 0.0, None, f, None, None, None)
assert rc == R.ERR_UNSUPPORTED, rc
assert b"scratch" in lib.rolekv_last_error()
# pooling without a pre-pool output buffer is refused too
small = R.BatchDesc(1, 1, 8, 2, 128, 1000, None, None)
rc = lib.snapkv_score_noalloc(ctypes.byref(small), t, t, 32, 7, 0.0, None, f, None, None, None)
assert rc == R.ERR_INVALID_ARG, rc
assert b"scores_prepool" in lib.rolekv_last_error()
# so is a missing output; an empty batch needs none
rc = lib.snapkv_score_noalloc(ctypes.byref(small), t, t, 32, 1, 0.0, None, None, None, None, None)
assert rc == R.ERR_INVALID_ARG, rc
empty = R.BatchDesc(1, 1, 8, 2, 128, 0, None, None)
rc = lib.snapkv_score_noalloc(ctypes.byref(empty), t, t, 32, 7, 0.0, None, None, None, None, None)
assert rc == R.OK, rc
print("ok")
'''


def test_noalloc_rejects_on_the_host(lib):
    """snapkv_score_noalloc refuses a batch larger than its static scratch and
    pooling without a pre-pool buffer before any CUDA call.  Run in a child
    process with every GPU hidden, so that even a validation regression could
    only fail a CUDA call (a wrong return code), never touch a device."""
    import subprocess
    import sys
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    out = subprocess.run([sys.executable, "-c", _NOALLOC_REJECTS, B.ROOT], env=env,
                         capture_output=True, text=True, timeout=300)
    assert out.returncode == 0, out.stderr[-2000:]
    assert out.stdout.strip().endswith("ok")
