"""Several host threads make the library's first calls at the same moment.

The per-device facts and the one-time kernel attributes are set up by the first
call on a device; calls from other threads at that moment must neither race nor
block. Run in a fresh interpreter so that these really are the process's first
calls, each thread on its own stream (ctypes releases the GIL during a call).
"""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

_CHILD = r"""
import threading
import torch
import __graft_entry__
__graft_entry__.build()
from paper_2608_25332_gb300 import provip as P

n = 8
scores = [torch.rand(4, 3000 + 7 * i, device="cuda:0") for i in range(n)]
streams = [torch.cuda.Stream() for _ in range(n)]
torch.cuda.synchronize()
P.lib()  # load the library (no call on the device yet)
out, errs = [None] * n, []
gate = threading.Barrier(n)

def run(i):
    try:
        gate.wait()
        with torch.cuda.stream(streams[i]):
            out[i] = P.provip_topk(scores[i], 50)
        streams[i].synchronize()
    except Exception as e:  # reported below
        errs.append(repr(e))

threads = [threading.Thread(target=run, args=(i,)) for i in range(n)]
for t in threads:
    t.start()
for t in threads:
    t.join(timeout=120)
assert not any(t.is_alive() for t in threads), "a thread is stuck"
assert not errs, errs
for i in range(n):
    ref = torch.sort(torch.topk(scores[i], 50, dim=1).indices, dim=1).values.to(torch.int32)
    assert torch.equal(out[i], ref), i
rc, bits = P.provip_device_status(clear=True)
assert rc == 0 and bits == 0, (rc, bits)
print("threads ok")
"""


def test_concurrent_first_calls_from_host_threads():
    r = subprocess.run([sys.executable, "-c", _CHILD], cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0 and "threads ok" in r.stdout, r.stdout[-2000:] + r.stderr[-3000:]
