"""The canary-checking build (-DKVM_DEBUG) on the GPU: a maintenance round
through it leaves every canary band intact and matches the oracle; a band
spoiled from the host (kvm_debug_poke_canary, no kernel involved) is
reported by kvm_check as KVM_E_DEVICE naming the buffer.  The debug library
runs in a child process (a process loads one libkvm)."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import sys
sys.path[:0] = [{root!r}, {tests!r}]
from harness import Pair
from workload import synth as W
from paper_2609_18935_gb300 import kvm
w = W.make_workload("tiny")
pair = Pair(w.shape, w.prefix_len, w.capacity(), 64, seed_index=w.index, prefix="refill")
span_cu, sb, se, tails = W.round_plan(w, 0, [w.prefix_len[0]])
errs = pair.run_round(span_cu, sb, se, tails, W.tail_inputs(w, 0, tails))
assert all(v <= 5e-3 for v in errs.values()), errs
pair.ctx.check()
pair.ctx.debug_poke_canary()
try:
    pair.ctx.check()
except kvm.KvmError as e:
    assert e.code == kvm.KVM_E_DEVICE and "canary" in str(e), str(e)
    print("canary reported:", e)
else:
    raise SystemExit("the spoiled canary was not reported")
"""


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_debug_build_round_and_canary_report():
    from paper_2609_18935_gb300 import build_lib
    lib = build_lib.build(debug=True)
    env = dict(os.environ, KVM_LIB=lib)
    r = subprocess.run([sys.executable, "-c", CHILD.format(root=ROOT, tests=os.path.join(ROOT, "tests"))],
                       capture_output=True, text=True, timeout=600, env=env)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-3000:]
    assert "canary reported" in r.stdout


def test_release_build_has_no_canaries():
    from harness import Pair
    from paper_2609_18935_gb300 import kvm
    from workload import synth as W
    pair = Pair(W.TINY, [10], [128], 64, seed_index=3)
    with pytest.raises(kvm.KvmError) as ei:
        pair.ctx.debug_poke_canary()
    assert ei.value.code == kvm.KVM_E_UNSUPPORTED
