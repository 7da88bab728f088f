"""The pruning step with its sequences in host memory (PROVIP_PRUNE_HOST_ROWS).

hidden, V and the position ids stay in pinned host memory mapped into the
GPU's address space, the compacted outputs are written there too, and only Q
and K are device memory. Every output must be bit-identical to the same call
with everything on the device (the selection is the same computation; the
compaction copies the same bytes by another route), for the LLaVA-NeXT and
video GQA workloads (bulk-sized and 1 KiB rows) and a ragged LLaVA-1.5 batch.
"""
import pytest
import torch

from paper_2608_25332_gb300 import provip as P
from paper_2608_25332_gb300 import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()
    yield
    rc, bits = P.provip_device_status(clear=True)
    assert rc == 0 and bits == 0, f"device status {rc} {bits}"


@pytest.mark.parametrize("name,batch", [("llava_next_7b_bf16_b8", 2), ("video_gqa_bf16_b1", None),
                                        ("llava15_7b_bf16_b16", 5)])
@pytest.mark.parametrize("flags", [0, P.PRUNE_OVERLAP_PREVIOUS])
def test_host_rows_match_device_rows(name, batch, flags):
    w = synth.BY_NAME[name]
    cpu = synth.in_llm_inputs(w, batch=batch)
    g = {k: (v.to(DEV) if isinstance(v, torch.Tensor) else v) for k, v in cpu.items()}
    hst = {k: cpu[k].pin_memory() for k in ("hidden", "V", "pos")}
    dev_step = P.PruneStep(g["Q"], g["K"], g["V"], g["hidden"], g["pos"], cpu["head_list"], w.n_t[1], g["N_v"],
                           g["keep"], want_scores=True, flags=flags)
    host_step = P.PruneStep(g["Q"], g["K"], hst["V"], hst["hidden"], hst["pos"], cpu["head_list"], w.n_t[1],
                            g["N_v"], g["keep"], want_scores=True, flags=flags, host_rows=True)
    assert not host_step.hidden_out.is_cuda and host_step.hidden_out.is_pinned()
    ref = dev_step(g["Q"], g["K"], g["V"], g["hidden"], g["pos"], g["text_start"], g["text_len"], g["seq_len"],
                   g["vis_start"])
    # twice in a row (the second call overwrites the first's outputs in place)
    for _ in range(2):
        got = host_step(g["Q"], g["K"], hst["V"], hst["hidden"], hst["pos"], g["text_start"], g["text_len"],
                        g["seq_len"], g["vis_start"])
    torch.cuda.synchronize()
    assert torch.equal(got["idx"], ref["idx"]) and torch.equal(got["seq_len"], ref["seq_len"])
    assert torch.equal(got["scores"], ref["scores"])
    slo = ref["seq_len"].cpu()
    for k in ("hidden", "K", "V"):
        for b in range(slo.shape[0]):
            n = int(slo[b])
            assert torch.equal(got[k][b, :n].view(torch.int16), ref[k][b, :n].cpu().view(torch.int16)), (k, b)
    for b in range(slo.shape[0]):
        n = int(slo[b])
        assert torch.equal(got["pos"][:, b, :n], ref["pos"][:, b, :n].cpu())


@pytest.mark.parametrize("name,batch", [("llava_next_7b_bf16_b8", 2), ("video_gqa_bf16_b1", None),
                                        ("llava15_7b_bf16_b16", 5)])
@pytest.mark.parametrize("outputs", ["device", "host"])
def test_compact_detects_host_memory(name, batch, outputs):
    """provip_compact with hidden, K, V and the position ids in pinned host
    memory (detected by the library), writing device or host outputs, gives the
    bytes of the all-device call."""
    w = synth.BY_NAME[name]
    cpu = synth.in_llm_inputs(w, batch=batch)
    g = {k: (v.to(DEV) if isinstance(v, torch.Tensor) else v) for k, v in cpu.items()}
    st = P.PruneStep(g["Q"], g["K"], g["V"], g["hidden"], g["pos"], cpu["head_list"], w.n_t[1], g["N_v"],
                     g["keep"], want_scores=False)
    idx = st(g["Q"], g["K"], g["V"], g["hidden"], g["pos"], g["text_start"], g["text_len"], g["seq_len"],
             g["vis_start"])["idx"].clone()
    ref = P.provip_compact(idx, g["hidden"], g["K"], g["V"], g["pos"], g["seq_len"], g["vis_start"], g["N_v"])
    hst = {k: cpu[k].pin_memory() for k in ("hidden", "K", "V", "pos")}
    out = None
    if outputs == "host":
        out = tuple(torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
                    for t in (ref["hidden"], ref["K"], ref["V"], ref["pos"]))
    got = P.provip_compact(idx, hst["hidden"], hst["K"], hst["V"], hst["pos"], g["seq_len"], g["vis_start"],
                           g["N_v"], out=out)
    torch.cuda.synchronize()
    assert torch.equal(got["seq_len"], ref["seq_len"])
    slo = ref["seq_len"].cpu()
    for k in ("hidden", "K", "V"):
        for b in range(slo.shape[0]):
            n = int(slo[b])
            assert torch.equal(got[k][b, :n].cpu().view(torch.int16), ref[k][b, :n].cpu().view(torch.int16)), (k, b)
    for b in range(slo.shape[0]):
        n = int(slo[b])
        assert torch.equal(got["pos"][:, b, :n].cpu(), ref["pos"][:, b, :n].cpu())
