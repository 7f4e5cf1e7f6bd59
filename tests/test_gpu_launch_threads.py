"""Launch set-up from several host threads: the dynamic shared-memory opt-in of each kernel is
recorded per (device, kernel) under a lock, so first calls made at the same moment from two
threads with different shared-memory sizes (different context lengths give different split
lengths) all launch, and give the outputs of the same calls made one at a time.  Runs in a fresh
process so that no opt-in has been made before the threads start."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SCRIPT = r"""
import sys, threading
sys.path.insert(0, sys.argv[1]); sys.path.insert(0, sys.argv[1] + "/tests")
import numpy as np, torch
import paper_2608_14191_gb300 as aatc
import harness as Hn
import workloads as W
aatc.load()
cfg = W.Config(8, "threads", 1, 2, 8, 1, 20000, (2.75,), 1, "two-thread first calls")
case = Hn.Case(aatc, cfg, 2.75, n_calib=1024)
kd, vd = W.kv_device(cfg, 0, 1, cfg.n_ctx, "cuda:0")
cache = case.plan.new_cache(1, cfg.n_ctx, "cuda:0")
aatc.encode(case.plan, 0, kd, vd, cache, 0, cfg.n_ctx)
q = W.queries_device(cfg, 0, 1, 1, "cuda:0")[0]
torch.cuda.synchronize()
ctxs = [20000, 700, 9000, 3000]
outs = {}
errors = []
bar = threading.Barrier(len(ctxs))
def run(n):
    try:
        torch.cuda.set_device(0)
        s = torch.cuda.Stream()
        bar.wait()
        with torch.cuda.stream(s):
            o = aatc.decode_attention(case.plan, 0, q, cache, n, cfg.n_ctx, stream=s)
        s.synchronize()
        outs[n] = o.cpu()
    except Exception as e:
        errors.append(repr(e))
ts = [threading.Thread(target=run, args=(n,)) for n in ctxs]
[t.start() for t in ts]
[t.join() for t in ts]
assert not errors, errors
for n in ctxs:
    again = aatc.decode_attention(case.plan, 0, q, cache, n, cfg.n_ctx).cpu()
    assert torch.equal(outs[n], again), n
assert case.plan.device_error() == 0
print("threads ok")
"""


def test_first_calls_from_four_threads():
    r = subprocess.run([sys.executable, "-c", SCRIPT, ROOT], capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    assert "threads ok" in r.stdout
