"""Several host threads make the library's first calls at the same moment.

The per-device facts and the one-time kernel set-up (kernel attributes, the
cluster form's placement checks, the address of the no-alloc scratch array)
are done by the first call that needs them; calls from other threads at that
moment must neither race nor block, and must take the same kernel form as a
call made alone. Each case runs in a fresh interpreter so that these really are
the process's first calls (ctypes releases the GIL during a call).
"""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

_PRELUDE = r"""
import threading
import torch
import __graft_entry__
__graft_entry__.build()
from paper_2608_25332_gb300 import provip as P
from paper_2608_25332_gb300 import synth

def run_threads(n, body):
    out, errs = [None] * n, []
    gate = threading.Barrier(n)
    def run(i):
        try:
            gate.wait()
            out[i] = body(i)
        except Exception as e:  # reported below
            errs.append(repr(e))
    threads = [threading.Thread(target=run, args=(i,)) for i in range(n)]
    for t in threads:
        t.start()
    for t in threads:
        t.join(timeout=300)
    assert not any(t.is_alive() for t in threads), "a thread is stuck"
    assert not errs, errs
    return out
"""

# eight threads, each on its own stream with its own workspace, whose first
# calls are the one-time set-up paths of the library: the cluster head-score
# form (three threads at once on the same kernel shape, plain and through
# ALGO_AUTO), the streaming and two-pass forms, the cluster form with the
# confidence statistics (visual heads), the pre-LLM pass and the top-k
_MIXED = _PRELUDE + r"""
w = synth.BY_NAME["llava15_7b_bf16_b16"]
dev = "cuda:0"
cpu = synth.in_llm_inputs(w, batch=2, with_kv=False)
cv = synth.in_llm_inputs(w, batch=2, with_kv=False, visual_heads=True)
pre = synth.pre_llm_inputs(w, batch=2)
g = {k: (v.to(dev) if isinstance(v, torch.Tensor) else v) for k, v in cpu.items()}
gv = {k: (v.to(dev) if isinstance(v, torch.Tensor) else v) for k, v in cv.items()}
gp = {k: v.to(dev) for k, v in pre.items()}
scores = torch.rand(4, 3000, device=dev)
streams = [torch.cuda.Stream() for _ in range(8)]
torch.cuda.synchronize()
P.lib()  # load the library (no call on the device yet)
Ntm = w.n_t[1]
hs = lambda algo: P.provip_head_scores(g["Q"], g["K"], g["head_list"], g["text_start"], g["text_len"],
                                       g["seq_len"], g["vis_start"], g["N_v"], algo=algo, N_t_max=Ntm)
calls = [
    lambda: hs(P.ALGO_TCGEN05_CLUSTER),
    lambda: hs(P.ALGO_TCGEN05_CLUSTER),
    lambda: hs(P.ALGO_AUTO),
    lambda: hs(P.ALGO_TCGEN05_STREAM),
    lambda: hs(P.ALGO_TCGEN05_TWOPASS),
    lambda: P.provip_head_confidence(gv["Q"], gv["K"], gv["text_start"], gv["text_len"], gv["seq_len"],
                                     gv["vis_start"], gv["N_v"], 6, algo=P.ALGO_TCGEN05_CLUSTER,
                                     N_t_max=Ntm)[1],
    lambda: P.provip_similarity_reduce(gp["emb_v"], gp["emb_t"], gp["text_len"], w.keep_pre)["merged"],
    lambda: P.provip_topk(scores, 50),
]

def body(i):
    with torch.cuda.stream(streams[i]):
        r = calls[i]()
    streams[i].synchronize()
    return r

got = run_threads(8, body)
for i in range(8):
    ref = calls[i]()  # the same call again, alone
    torch.cuda.synchronize()
    assert torch.equal(got[i], ref), f"call {i} differs from the same call made alone"
rc, bits = P.provip_device_status(clear=True)
assert rc == 0 and bits == 0, (rc, bits)
print("threads ok")
"""

# eight threads make their first no-alloc call at the same instant. They share
# one stream, so their kernels run one after another on the GPU (calls that
# overlap on the GPU race on the shared scratch by design); identical inputs
# make every interleaving of the enqueued kernels give the same bits.
_NOALLOC = _PRELUDE + r"""
w = synth.BY_NAME["llava15_7b_bf16_b16"]
dev = "cuda:0"
cpu = synth.in_llm_inputs(w, batch=2, with_kv=False)
g = {k: (v.to(dev) if isinstance(v, torch.Tensor) else v) for k, v in cpu.items()}
shared = torch.cuda.Stream()
torch.cuda.synchronize()
P.lib()
args = (g["Q"], g["K"], g["head_list"], g["text_start"], g["text_len"], g["seq_len"], g["vis_start"],
        g["N_v"])

def body(i):
    with torch.cuda.stream(shared):
        return P.provip_head_scores_noalloc(*args, algo=P.ALGO_TCGEN05_CLUSTER, N_t_max=w.n_t[1])

got = run_threads(8, body)
shared.synchronize()
ref = P.provip_head_scores(*args, algo=P.ALGO_TCGEN05_CLUSTER, N_t_max=w.n_t[1])
torch.cuda.synchronize()
for i in range(8):
    assert torch.equal(got[i], ref), f"no-alloc call {i} differs from provip_head_scores"
rc, bits = P.provip_device_status(clear=True)
assert rc == 0 and bits == 0, (rc, bits)
print("threads ok")
"""


def _run(child):
    r = subprocess.run([sys.executable, "-c", child], cwd=ROOT, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0 and "threads ok" in r.stdout, r.stdout[-2000:] + r.stderr[-3000:]


def test_concurrent_first_calls_of_every_one_time_setup():
    _run(_MIXED)


def test_concurrent_first_noalloc_calls():
    _run(_NOALLOC)
