"""Back-to-back pre-LLM passes (Sec. 4.2-4.3) on one workspace and one stream.

The pass chains its kernels as programmatic dependents (each waits for the
kernels before it only where it reads what they wrote), and consecutive passes
share the workspace (the permuted copy, the argmax partials, the sort's lists).
Three passes over alternating batches, enqueued with no synchronisation between
them, eagerly and replayed from one CUDA graph, must each give exactly the
outputs of the same batch run on its own with a fresh workspace: the keep set,
the assignment, the merged rows and p, bit for bit."""
import numpy as np
import pytest
import torch

from paper_2608_25332_gb300 import provip as P

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()
    yield
    rc, bits = P.provip_device_status(clear=True)
    assert rc == 0 and bits == 0, f"device status {rc} {bits}"


def _batch(seed, B, N_v, D, N_t):
    g = torch.Generator().manual_seed(seed)
    ev = torch.randn(B, N_v, D, generator=g).to(torch.bfloat16)
    et = (torch.randn(B, N_t, D, generator=g) * (0.25 / D ** 0.25)).to(torch.bfloat16)
    tl = torch.randint(1, N_t + 1, (B,), generator=g, dtype=torch.int32)
    return ev.to(DEV), et.to(DEV), tl.to(DEV)


def _outputs(B, N_v, D, N_t, keep):
    return dict(idx=torch.empty(B, keep, dtype=torch.int32, device=DEV),
                merged=torch.empty(B, keep, D, dtype=torch.bfloat16, device=DEV),
                p=torch.empty(B, N_v, dtype=torch.float32, device=DEV),
                mask=torch.empty(B, N_t, dtype=torch.uint8, device=DEV),
                assign=torch.empty(B, N_v, dtype=torch.int32, device=DEV))


def _same(a, b, what):
    for k in ("idx", "assign", "merged", "p", "mask"):
        assert torch.equal(a[k], b[k]), f"{what}: {k} differs"


@pytest.mark.parametrize("B,N_v,D,N_t,keep", [
    (4, 576, 256, 48, 192),     # LLaVA-1.5-like: one 512-row group of pruned rows per sample
    (2, 2880, 512, 96, 960),    # anyres-like: four groups, the pair Gram's mixed column ranges
])
def test_back_to_back_passes_match_single_runs(B, N_v, D, N_t, keep):
    X, Y = _batch(11, B, N_v, D, N_t), _batch(12, B, N_v, D, N_t)
    ref = []
    for ev, et, tl in (X, Y):
        o = _outputs(B, N_v, D, N_t, keep)
        P.provip_similarity_reduce(ev, et, tl, keep, want_merged=True, out=o)
        torch.cuda.synchronize()
        ref.append({k: v.clone() for k, v in o.items()})
    need = P.lib().provip_similarity_reduce_workspace_size(B, N_v, D, N_t, keep)
    ws = P.workspace(need, torch.device(DEV))
    outs = [_outputs(B, N_v, D, N_t, keep) for _ in range(3)]
    batches = (X, Y, X)

    def chain():
        for (ev, et, tl), o in zip(batches, outs):
            P.provip_similarity_reduce(ev, et, tl, keep, want_merged=True, out=o, ws=ws)

    chain()
    torch.cuda.synchronize()
    for i, o in enumerate(outs):
        _same(o, ref[i % 2], f"eager pass {i}")
    for o in outs:
        for v in o.values():
            v.zero_()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        chain()
    g.replay()
    g.replay()
    torch.cuda.synchronize()
    for i, o in enumerate(outs):
        _same(o, ref[i % 2], f"graph pass {i}")
