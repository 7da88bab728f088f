"""The head-scores entry point that allocates nothing, against the regular one.

provip_head_scores_noalloc is for hosts that cannot give the library any
device memory (a framework that owns every allocation and passes only tensors,
or a serving loop that bans allocator calls); its scratch is a static array in
the library. Two calls in a row, on different workloads, must each match
provip_head_scores on the same inputs within the parity tolerance, so stale
contents left in the shared array by the first call cannot leak into the second.
This file is collected last so that a failure here stops a -x run only after
every other test has run.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_25332_gb300 import provip as P
from paper_2608_25332_gb300 import synth
from parity import assert_close_rel, rtol_for

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()


def _inputs(name, batch=None):
    w = synth.BY_NAME[name]
    cpu = synth.in_llm_inputs(w, batch=batch, with_kv=False)
    return w, {k: (v.to(DEV) if isinstance(v, torch.Tensor) else v) for k, v in cpu.items()}


def _both(w, g, algo):
    args = (g["Q"], g["K"], g["head_list"], g["text_start"], g["text_len"], g["seq_len"], g["vis_start"],
            g["N_v"])
    ref = P.provip_head_scores(*args, algo=algo, N_t_max=w.n_t[1])
    got = P.provip_head_scores_noalloc(*args, algo=algo, N_t_max=w.n_t[1])
    torch.cuda.synchronize()
    return ref.cpu().numpy(), got.cpu().numpy()


def test_noalloc_matches_workspace_version_twice():
    # first call: LLaVA-1.5-7B shapes, ragged text lengths; second: the video GQA
    # workload (different shape, so the shared scratch holds the first call's data);
    # then the same LLaVA-1.5 shapes with the streaming and two-pass tcgen05
    # forms forced (the tiny batch would otherwise take the cluster form) and the
    # CUDA-core form, so that every kernel form that uses the scratch is checked
    # against the workspace version
    for name, batch, algo in (("llava15_7b_bf16_b16", 4, P.ALGO_AUTO), ("video_gqa_bf16_b1", None, P.ALGO_AUTO),
                              ("llava15_7b_bf16_b16", 4, P.ALGO_TCGEN05_STREAM),
                              ("llava15_7b_bf16_b16", 4, P.ALGO_TCGEN05_TWOPASS),
                              ("llava15_7b_bf16_b16", 4, P.ALGO_SIMT)):
        w, g = _inputs(name, batch)
        ref, got = _both(w, g, algo)
        assert_close_rel(got, ref, rtol_for(w.dtype), f"noalloc {name} algo={algo}")
    rc, bits = P.provip_device_status(clear=True)
    assert rc == 0 and bits == 0


def test_noalloc_rejects_shapes_beyond_the_static_scratch():
    # B=64, L_max=4096, 64 heads: several hundred MB of scratch, far above 4 MiB
    L = P.lib()
    need = L.provip_head_scores_workspace_size(64, 4096, 64, 128, 2048, P.ALGO_TCGEN05, P.BF16)
    assert need > (4 << 20)
    heads = (ctypes.c_int * 64)(*range(64))
    fake = ctypes.c_void_p(0x10000)
    rc = L.provip_head_scores_noalloc(fake, fake, 64, 4096, 64, 64, 128, heads, 64, fake, fake, None, 128,
                                      100, 2048, fake, P.BF16, P.ALGO_TCGEN05, fake, None)
    assert rc == P.ERR_UNSUPPORTED
    assert b"static array" in L.provip_last_error()
