"""The selection (head scores + top-k, Sec. 4.4) and the pruning step under
the ways a caller reuses buffers and streams.

Every selection is compared bit for bit with the stand-alone score reduction
followed by the stand-alone top-k, which share its arithmetic:
  * a workspace full of random bytes (the header promises that the workspace
    needs no initialisation), then further calls on what the first one left;
  * CUDA graphs holding one and three calls, replayed several times;
  * two shapes taking turns on one workspace;
  * overlapped calls (PROVIP_PRUNE_OVERLAP_PREVIOUS) of the whole pruning step
    with a row mask, against serial calls;
  * overlapped calls sharing one idx buffer: a call's top-k may only rewrite
    idx once the previous call's compaction has read it (the head-score kernel
    holds its completion for that), for the cluster and the streaming forms.
"""
import pytest
import torch

from paper_2608_25332_gb300 import provip as P
from paper_2608_25332_gb300 import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
NAMES = ["llava_next_7b_bf16_b8", "video_gqa_bf16_b1", "llava15_7b_bf16_b16"]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()
    yield
    rc, bits = P.provip_device_status(clear=True)
    assert rc == 0 and bits == 0, f"device status {rc} {bits}"


_cache = {}


def inputs(name, seed_shift=0):
    key = (name, seed_shift)
    if key not in _cache:
        w = synth.BY_NAME[name]
        cpu = synth.in_llm_inputs(w, seed=w.seed + seed_shift)
        _cache[key] = (w, {k: (v.to(DEV) if isinstance(v, torch.Tensor) else v) for k, v in cpu.items()})
    return _cache[key]


def reference(w, g, row_mask=None):
    s = P.provip_head_scores(g["Q"], g["K"], g["head_list"], g["text_start"], g["text_len"], g["seq_len"],
                             g["vis_start"], g["N_v"], row_mask=row_mask, algo=P.ALGO_TCGEN05_CLUSTER,
                             N_t_max=w.n_t[1])
    return P.provip_topk(s, g["keep"]), s


def selection(w, g, ws, row_mask=None):
    return P.provip_head_topk(g["Q"], g["K"], g["head_list"], g["text_start"], g["text_len"], g["seq_len"],
                              g["vis_start"], g["N_v"], g["keep"], row_mask=row_mask,
                              algo=P.ALGO_TCGEN05_CLUSTER, N_t_max=w.n_t[1], ws=ws)


def ws_for(w, g):
    n = P.lib().provip_head_scores_workspace_size(w.B, w.L_max, w.H_sel, w.n_t[1], g["N_v"],
                                                  P.ALGO_TCGEN05_CLUSTER, P.BF16)
    return P.workspace(n, DEV)


@pytest.mark.parametrize("name", NAMES)
def test_random_workspace(name):
    w, g = inputs(name)
    ref_idx, ref_s = reference(w, g)
    ws = ws_for(w, g)
    gen = torch.Generator(device=DEV).manual_seed(1234)
    for rep in range(3):
        ws.copy_(torch.randint(0, 256, ws.shape, dtype=torch.uint8, device=DEV, generator=gen))
        # the first call on random bytes, the next ones on what it left
        for call in range(3):
            idx, s = selection(w, g, ws)
            torch.cuda.synchronize()
            assert torch.equal(s, ref_s), (name, rep, call)
            assert torch.equal(idx, ref_idx), (name, rep, call)


@pytest.mark.parametrize("calls", [1, 3])
@pytest.mark.parametrize("name", ["llava_next_7b_bf16_b8", "video_gqa_bf16_b1"])
def test_graph_replays(name, calls):
    w, g = inputs(name)
    ref_idx, ref_s = reference(w, g)
    ws = ws_for(w, g)
    ws.fill_(0xA5)
    idx = torch.empty((w.B, g["keep"]), dtype=torch.int32, device=DEV)
    scores = torch.empty((w.B, g["N_v"]), dtype=torch.float32, device=DEV)
    heads, hs = P._heads_arg(g["head_list"], w.H_q)
    L = P.lib()

    def call():
        rc = L.provip_head_topk(P._ptr(g["Q"]), P._ptr(g["K"]), w.B, w.L_max, w.H_q, w.H_kv, 128, heads, hs,
                                P._i32(g["text_start"]), P._i32(g["text_len"]), None, w.n_t[1], g["vis_start"],
                                g["N_v"], P._i32(g["seq_len"]), g["keep"], P.BF16, P.ALGO_TCGEN05_CLUSTER,
                                P._ptr(idx), P._ptr(scores), P._ptr(ws), ws.numel(), P._stream(DEV))
        assert rc == 0

    s = torch.cuda.Stream(device=DEV)
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        call()  # warm-up outside the capture (one-time kernel attributes)
    s.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        for _ in range(calls):
            call()
    for rep in range(4):
        idx.fill_(-1)
        scores.fill_(float("nan"))
        graph.replay()
        torch.cuda.synchronize()
        assert torch.equal(idx, ref_idx), (name, calls, rep)
        assert torch.equal(scores, ref_s), (name, calls, rep)


def test_two_shapes_share_a_workspace():
    wa, ga = inputs("llava_next_7b_bf16_b8")
    wb, gb = inputs("llava15_7b_bf16_b16")
    ra, rb = reference(wa, ga)[0], reference(wb, gb)[0]
    n = max(ws_for(wa, ga).numel(), ws_for(wb, gb).numel())
    ws = P.workspace(n, DEV)
    for rep in range(3):
        ia, _ = selection(wa, ga, ws)
        ib, _ = selection(wb, gb, ws)
        torch.cuda.synchronize()
        assert torch.equal(ia, ra) and torch.equal(ib, rb), rep


@pytest.mark.parametrize("name", ["llava_next_7b_bf16_b8", "video_gqa_bf16_b1"])
def test_overlapped_steps_with_row_mask(name):
    """The whole step, overlapped, with a row mask, against serial calls and
    against the stand-alone selection."""
    w, g0 = inputs(name)
    batches = [g0, inputs(name, 91)[1], inputs(name, 92)[1]]
    gen = torch.Generator().manual_seed(7)
    masks = [(torch.rand((w.B, w.n_t[1]), generator=gen) > 0.3).to(torch.uint8).to(DEV) for _ in batches]
    ws = P.workspace(P.lib().provip_prune_workspace_size(w.B, w.L_max, w.H_sel, w.n_t[1], g0["N_v"],
                                                         P.ALGO_TCGEN05_CLUSTER, P.BF16), DEV)

    def run(flags, sync):
        outs = []
        for c, m in zip(batches, masks):
            st = P.PruneStep(c["Q"], c["K"], c["V"], c["hidden"], c["pos"], c["head_list"], w.n_t[1], c["N_v"],
                             c["keep"], algo=P.ALGO_TCGEN05_CLUSTER, flags=flags, ws=ws)
            outs.append(st(c["Q"], c["K"], c["V"], c["hidden"], c["pos"], c["text_start"], c["text_len"],
                           c["seq_len"], c["vis_start"], m))
            if sync:
                torch.cuda.synchronize()
        torch.cuda.synchronize()
        return [{k: v.clone() for k, v in o.items() if v is not None} for o in outs]

    serial = run(0, True)
    for c, m, o in zip(batches, masks, serial):
        ref_idx, ref_s = reference(w, c, row_mask=m)
        assert torch.equal(o["idx"], ref_idx) and torch.equal(o["scores"], ref_s)
    for rep in range(3):
        over = run(P.PRUNE_OVERLAP_PREVIOUS, False)
        for a, b in zip(serial, over):
            for k in a:
                assert torch.equal(a[k], b[k]), f"overlapped call differs in {k} (rep {rep})"


@pytest.mark.parametrize("algo", ["ALGO_TCGEN05_CLUSTER", "ALGO_TCGEN05_STREAM"])
@pytest.mark.parametrize("name", ["llava_next_7b_bf16_b8", "video_gqa_bf16_b1"])
def test_overlap_with_one_idx_buffer(name, algo):
    """Overlapped calls that share one idx buffer and one workspace but write
    their rows to separate outputs: a selection that rewrote idx while the
    previous call's compaction still read it would show up as rows of the
    wrong batch in that call's outputs."""
    algo = getattr(P, algo)
    w, g0 = inputs(name)
    batches = [g0, inputs(name, 91)[1], inputs(name, 92)[1]]
    st = P.PruneStep(g0["Q"], g0["K"], g0["V"], g0["hidden"], g0["pos"], g0["head_list"], w.n_t[1], g0["N_v"],
                     g0["keep"], algo=algo, want_scores=False, flags=P.PRUNE_OVERLAP_PREVIOUS)
    outs = [tuple(torch.empty_like(t) for t in (st.hidden_out, st.K_out, st.V_out, st.pos_out)) for _ in batches]

    def run(sync):
        res = []
        for c, o in zip(batches, outs):
            st.hidden_out, st.K_out, st.V_out, st.pos_out = o
            r = st(c["Q"], c["K"], c["V"], c["hidden"], c["pos"], c["text_start"], c["text_len"], c["seq_len"],
                   c["vis_start"])
            if sync:
                torch.cuda.synchronize()
                res.append(r["idx"].clone())
        torch.cuda.synchronize()
        return res, [tuple(t.clone() for t in o) for o in outs]

    ref_idx, ref_rows = run(True)
    for rep in range(5):
        for o in outs:
            for t in o:
                t.zero_()
        _, rows = run(False)
        assert torch.equal(st.idx, ref_idx[-1]), rep
        for i, (a, b) in enumerate(zip(ref_rows, rows)):
            for k, (x, y) in enumerate(zip(a, b)):
                assert torch.equal(x, y), f"call {i} output {k} differs (rep {rep})"
