"""The paper's progressive pruning schedule (Sec. 4.1) on one stream, with no
host synchronisation between the stages (and the ablation of Sec. 5 without
the pre-LLM stage):

  1. before the LLM (Sec. 4.2-4.3): N_v -> N1 visual tokens by text-guided
     similarity, pruned tokens merged into their nearest kept token;
  2. at the shallow pruning layer (Sec. 4.4, visual heads only): the N_vis most
     confident heads of each sample (confidence over the critical text rows T
     found in stage 1), N1 -> N2 by their attention, sequence compacted;
  3. at the middle pruning layer (Sec. 4.4, all attention heads): N2 -> N3 by
     the attention of every head over the compacted sequence.

Every stage is one call of the C ABI (provip_similarity_reduce,
provip_prune_visual_heads, provip_prune); this module only owns the device
buffers that carry one stage's outputs into the next (the T mask, the
compacted keys/values/hidden states/position ids and sequence lengths), so a
whole schedule can be captured in one CUDA graph. The LLM layers between the
stages are not part of this library: the caller hands each pruning layer the
queries (and, for the shallow layer, keys/values/hidden states) its layer
computed.
"""
from __future__ import annotations

import torch

from . import provip as P


class ProgressiveSchedule:
    """Buffers and workspaces of one schedule shape.

    B samples; N_v visual tokens of dimension D_v before the LLM; text rows
    N_t_max; the shallow layer sees L1 = L_max rows (vis_start system rows,
    N1 visual rows, the text) with H_q/H_kv heads of 128 and hidden size D;
    keeps N1, N2, N3 visual tokens after the three stages; N_vis visual heads.
    """

    def __init__(self, B, N_v, D_v, N_t_max, L_max, H_q, H_kv, D, P_ids, N1, N2, N3, N_vis,
                 dtype=torch.bfloat16, device="cuda", algo=P.ALGO_AUTO, pre_llm=True,
                 shallow_heads="visual"):
        """pre_llm=False: the ablation without pruning before the LLM (N1 = N_v;
        the critical text rows T are still found, by provip_crit_text).
        shallow_heads: "visual" (the N_vis most confident heads of each sample)
        or "all" (every head) at the shallow layer."""
        if not pre_llm and N1 != N_v:
            raise ValueError("without pre-LLM pruning N1 must equal N_v")
        if shallow_heads not in ("visual", "all"):
            raise ValueError("shallow_heads is 'visual' or 'all'")
        self.B, self.N_v, self.N_t_max, self.L_max = B, N_v, N_t_max, L_max
        self.N1, self.N2, self.N3, self.N_vis, self.algo = N1, N2, N3, N_vis, algo
        self.pre_llm, self.shallow_heads = pre_llm, shallow_heads
        dev = torch.device(device)
        L = P.lib()
        self.idx1 = torch.empty((B, N1), dtype=torch.int32, device=dev) if pre_llm else None
        self.merged = torch.empty((B, N1, D_v), dtype=dtype, device=dev) if pre_llm else None
        self.p = torch.empty((B, N_v), dtype=torch.float32, device=dev) if pre_llm else None
        self.mask = torch.empty((B, N_t_max), dtype=torch.uint8, device=dev)
        self.ws_pre = P.workspace(
            L.provip_similarity_reduce_workspace_size(B, N_v, D_v, N_t_max, N1) if pre_llm
            else L.provip_crit_text_workspace_size(B, N_t_max, D_v), dev)
        # shallow layer: outputs of provip_prune_visual_heads (shapes given by
        # meta tensors; the buffers live on dev)
        Q1 = torch.empty((B, L_max, H_q, 128), dtype=dtype, device="meta")
        K1 = torch.empty((B, L_max, H_kv, 128), dtype=dtype, device="meta")
        H1 = torch.empty((B, L_max, D), dtype=dtype, device="meta")
        pos1 = torch.empty((P_ids, B, L_max), dtype=torch.int32, device="meta")
        if shallow_heads == "visual":
            self.shallow = P.VisualHeadsPruneStep(Q1, K1, K1, H1, pos1, N_t_max, N1, N2, N_vis, algo=algo,
                                                  device=dev)
        else:
            self.shallow = P.PruneStep(Q1, K1, K1, H1, pos1, None, N_t_max, N1, N2, algo=algo, device=dev)
        # middle layer: every head over the compacted sequence
        L2 = L_max - N1 + N2
        Q2 = torch.empty((B, L2, H_q, 128), dtype=dtype, device="meta")
        K2 = torch.empty((B, L2, H_kv, 128), dtype=dtype, device="meta")
        H2 = torch.empty((B, L2, D), dtype=dtype, device="meta")
        pos2 = torch.empty((P_ids, B, L2), dtype=torch.int32, device="meta")
        self.middle = P.PruneStep(Q2, K2, K2, H2, pos2, None, N_t_max, N2, N3, algo=algo, device=dev)

    def __call__(self, emb_v, emb_t, text_len, shallow, middle, vis_start):
        """Enqueues the three stages on the current stream.

        shallow: dict(Q, K, V, hidden, pos, text_start, seq_len) of the shallow
        pruning layer (L_max rows); middle: dict(Q, text_start) of the middle
        pruning layer (L_max - N1 + N2 rows; its keys, values, hidden states,
        position ids and lengths are the shallow layer's compacted outputs).
        Returns the outputs of every stage (device tensors owned by self)."""
        if self.pre_llm:
            pre = P.provip_similarity_reduce(emb_v, emb_t, text_len, self.N1, ws=self.ws_pre,
                                             out=dict(idx=self.idx1, merged=self.merged, p=self.p,
                                                      mask=self.mask))
        else:
            P.provip_crit_text(emb_t, text_len, out=self.mask, ws=self.ws_pre)
            pre = dict(mask=self.mask)
        s = shallow
        if self.shallow_heads == "visual":
            o1 = self.shallow(s["Q"], s["K"], s["V"], s["hidden"], s["pos"], s["text_start"], text_len,
                              s["seq_len"], vis_start, crit_mask=self.mask)
        else:
            o1 = self.shallow(s["Q"], s["K"], s["V"], s["hidden"], s["pos"], s["text_start"], text_len,
                              s["seq_len"], vis_start)
        o2 = self.middle(middle["Q"], o1["K"], o1["V"], o1["hidden"], o1["pos"], middle["text_start"],
                         text_len, o1["seq_len"], vis_start)
        return dict(pre=pre, shallow=o1, middle=o2)
