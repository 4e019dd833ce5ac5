"""The checked build on the GPU (librolekv_checked.so, -DROLEKV_CHECKED).

There every kernel checks each global access whose address it computes from
run-time data against the extent the call's shapes give the buffer; a miss
is skipped and sets STATUS_BOUNDS.  Both tests run the checked library in a
child process (ROLEKV_CHECKED=1 picks it), so this process keeps the plain
one:
- the kernel parity suites pass unchanged on it (a check that fired would
  have skipped an access and changed an output, or set the status word that
  those tests require to be 0);
- its extent self-test, which makes kv_compact's checks on the last rows fire
  while every access stays inside the real buffer, skips exactly those rows
  and reports STATUS_BOUNDS.
"""

import os
import subprocess
import sys

import pytest

from paper_2607_13205_gb300 import build as B

ROOT = B.ROOT

pytestmark = pytest.mark.gpu


def _checked_env():
    if not os.path.exists(B.CHECKED_LIB_PATH):
        B.build(checked=True)
    env = dict(os.environ)
    env["ROLEKV_CHECKED"] = "1"
    return env


def test_parity_suites_pass_on_the_checked_build():
    r = subprocess.run([sys.executable, "-m", "pytest", "tests/test_gpu_kernels.py", "tests/test_gpu_fuzz.py",
                        "-m", "gpu", "-x", "-q", "-p", "no:cacheprovider"],
                       cwd=ROOT, env=_checked_env(), capture_output=True, text=True, timeout=1200)
    tail = (r.stdout + r.stderr)[-3000:]
    assert r.returncode == 0, tail
    assert " passed" in r.stdout, tail


_SELFTEST = r"""
import torch
from paper_2607_13205_gb300 import inputs as I
from paper_2607_13205_gb300 import rolekv as R

assert R.checked_build(), "the child did not load the checked library"
dev = torch.device("cuda:0")
w = I.WORKLOADS["tiny"]
roles_np = I.workload_roles(w, seed=0)
K, V = I.make_kv(w, roles_np, seed=0, device=dev)
batch = R.Batch(w.L, w.b, w.Hq, w.Hkv, w.d, w.n)
B = 0.25
g = torch.Generator(device="cpu").manual_seed(7)
n_units = w.L * w.b * w.Hkv
keep = torch.stack([torch.sort(torch.randperm(w.n, generator=g)[:R.kept_count(w.n, B)]).values
                    for _ in range(n_units)]).to(torch.int32).reshape(batch.kept_shape(B)).to(dev)

def compact(shrink):
    k_out = torch.full(R.compact_shape(batch, B), 7.0, dtype=torch.bfloat16, device=dev)
    v_out = torch.full_like(k_out, 7.0)
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    if shrink:
        R.selftest_shrink_extent(shrink)
    R.kv_compact(batch, K, V, keep, B, k_out, v_out, status=st)
    torch.cuda.synchronize()
    return k_out.reshape(-1, w.d), v_out.reshape(-1, w.d), int(st.item())

ka, va, sa = compact(0)
kb, vb, sb = compact(3)
assert sa == 0, f"plain call status {sa}"
assert sb & R.STATUS_BOUNDS, f"shrunk call status {sb}"
assert torch.equal(ka[:-3], kb[:-3]) and torch.equal(va[:-3], vb[:-3]), "rows before the shrunk extent differ"
assert bool((kb[-3:].float() == 7.0).all()) and bool((vb[-3:].float() == 7.0).all()), \
    "rows past the shrunk extent were written"
assert not torch.equal(ka[-3:], kb[-3:]), "the skipped rows should differ from the written ones"
ka2, va2, sa2 = compact(0)                          # the arming was used up
assert sa2 == 0 and torch.equal(ka2, ka) and torch.equal(va2, va)
print("checked selftest ok")
"""


def test_checked_build_skips_and_reports_out_of_extent_rows():
    r = subprocess.run([sys.executable, "-c", _SELFTEST], cwd=ROOT, env=_checked_env(),
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, (r.stdout + r.stderr)[-3000:]
    assert "checked selftest ok" in r.stdout
