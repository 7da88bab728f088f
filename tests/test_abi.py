"""The C-ABI library builds, loads and exports every declared symbol, and its
host-side argument validation rejects bad calls before touching a GPU.

These run without a GPU: every call below fails validation (or only queries a
workspace size), which happens on the host before any CUDA call.
"""
import ctypes
import os
import re

import pytest

from paper_2608_25332_gb300 import build as pbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "provip.h")

FAKE = ctypes.c_void_p(0x10000)  # never dereferenced: validation fails first


@pytest.fixture(scope="module")
def L():
    pbuild.build()
    from paper_2608_25332_gb300 import provip
    return provip.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(provip_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("provip_similarity_reduce", "provip_head_scores", "provip_topk_compact", "provip_prune",
              "provip_crit_text", "provip_relevance", "provip_topk", "provip_merge", "provip_compact"):
        assert n in names


def test_library_exports_every_declared_symbol(L):
    raw = ctypes.CDLL(pbuild.LIB)
    missing = [n for n in declared_functions() if not hasattr(raw, n)]
    assert not missing, missing


def test_binding_signatures_cover_the_header():
    from paper_2608_25332_gb300 import provip
    assert sorted(provip._SIGS) == declared_functions()


def test_status_strings_and_version(L):
    assert L.provip_status_string(0) == b"PROVIP_OK"
    assert L.provip_status_string(-3) == b"PROVIP_ERR_WORKSPACE"
    assert L.provip_version() >= 10000


def test_set_option_validation(L):
    assert L.provip_set_option(1, 0) == 0  # PROVIP_OPT_MERGE_PAIRS off ...
    assert L.provip_set_option(1, 1) == 0  # ... and back to the default
    assert L.provip_set_option(1, 2) == -1
    assert L.provip_set_option(99, 1) == -1


def _heads(*h):
    return (ctypes.c_int * len(h))(*h)


def test_head_scores_validation(L):
    hs = lambda heads, n, **kw: L.provip_head_scores(
        FAKE, FAKE, kw.get("B", 2), kw.get("L", 100), kw.get("Hq", 8), kw.get("Hkv", 4), kw.get("dh", 128),
        heads, n, FAKE, FAKE, None, 16, 10, 50, FAKE, kw.get("dtype", 1), kw.get("algo", 0), FAKE, None, 0, None)
    assert hs(_heads(0, 9), 2) == -1          # head out of range
    assert hs(_heads(3, 3), 2) == -1          # duplicate head
    assert hs(_heads(0), 0) == -1             # no head
    assert hs(_heads(0), 1, Hkv=3) == -1      # Hq % Hkv != 0
    assert hs(_heads(0), 1, dh=64) == -2      # unsupported head dim
    assert hs(_heads(0), 1, dtype=0, algo=2) == -2  # tcgen05 path needs bf16
    assert hs(_heads(0), 1, L=40) == -1       # visual range past L_max
    assert hs(_heads(0, 1), 2) == -3          # workspace too small
    assert b"workspace" in L.provip_last_error()


def test_all_heads_null_list_validation(L):
    hs = lambda heads, n, Hq=8: L.provip_head_scores(
        FAKE, FAKE, 2, 100, Hq, 4, 128, heads, n, FAKE, FAKE, None, 16, 10, 50, FAKE, 1, 0, FAKE, None, 0, None)
    assert hs(None, 4) == -1                  # a NULL list means every head: needs H_sel == H_q
    assert hs(None, 8) == -3                  # accepted; only the workspace is missing
    assert hs(None, 72, Hq=72) == -1          # more than 64 heads


def test_visual_heads_validation(L):
    conf = lambda nvis, **kw: L.provip_head_confidence(
        FAKE, FAKE, 2, 100, kw.get("Hq", 8), 4, 128, FAKE, FAKE, None, 16, 10, 50, FAKE, nvis, 1, 0, None,
        kw.get("out", FAKE), None, 0, None)
    assert conf(0) == -1                      # N_vis < 1
    assert conf(9) == -1                      # N_vis > H_q
    assert conf(2, Hq=72) == -2               # more than 64 heads
    assert conf(2, out=None) == -1            # vis_heads_out is required
    assert conf(2) == -3                      # workspace too small
    need = L.provip_visual_heads_workspace_size(2, 100, 8, 16, 50, 2, 0, 1)
    assert need > L.provip_head_scores_workspace_size(2, 100, 8, 16, 50, 0, 1)
    prune = lambda keep, flags=0: L.provip_prune_visual_heads(
        FAKE, FAKE, FAKE, FAKE, 2, 100, 8, 4, 128, 64, FAKE, FAKE, None, 16, 10, 50, FAKE, None, 0, 2, keep,
        1, 0, FAKE, FAKE, FAKE, None, FAKE, None, None, None, None, None, 0, flags, None)
    assert prune(0) == -1                     # keep < 1
    assert prune(51) == -1                    # keep > N_v
    assert prune(5, flags=8) == -1            # unknown flag
    assert prune(5) == -3                     # workspace too small


def test_topk_and_compact_validation(L):
    assert L.provip_topk(FAKE, 1, 10, 0, FAKE, None) == -1
    assert L.provip_topk(FAKE, 1, 10, 11, FAKE, None) == -1
    assert L.provip_topk(FAKE, 1, 60000, 5, FAKE, None) == -2
    # keep > N_v
    assert L.provip_compact(FAKE, 1, 10, 11, FAKE, 64, None, None, 0, 0, None, 0, FAKE, 50, 5, 1,
                            FAKE, None, None, None, None, None) == -1
    # K without K_out
    assert L.provip_compact(FAKE, 1, 10, 5, FAKE, 64, FAKE, None, 4, 128, None, 0, FAKE, 50, 5, 1,
                            FAKE, None, None, None, None, None) == -1
    # row bytes not a multiple of 16 (D = 4 bf16 = 8 bytes)
    assert L.provip_compact(FAKE, 1, 10, 5, FAKE, 4, None, None, 0, 0, None, 0, FAKE, 50, 5, 1,
                            FAKE, None, None, None, None, None) == -2
    # misaligned pointer
    assert L.provip_compact(FAKE, 1, 10, 5, ctypes.c_void_p(0x10008), 64, None, None, 0, 0, None, 0,
                            FAKE, 50, 5, 1, FAKE, None, None, None, None, None) == -2


def test_similarity_validation(L):
    assert L.provip_crit_text(FAKE, 1, 16, 12, FAKE, 1, FAKE, None, None, 0, None) == -2  # D % 8
    assert L.provip_merge(FAKE, 1, 10, 64, FAKE, 11, 1, FAKE, None, None, 0, None) == -1  # keep > N_v
    assert L.provip_merge(FAKE, 1, 10, 16384, FAKE, 5, 1, FAKE, FAKE, None, 0, None) == -2  # D > 8192
    assert L.provip_similarity_reduce(FAKE, 1, 10, 64, FAKE, FAKE, 8, None, 0, 1, FAKE, None, None, None,
                                      None, None, 0, None) == -1  # keep_pre = 0
    assert L.provip_relevance(FAKE, 1, 10, 64, FAKE, FAKE, 8, FAKE, 1, FAKE, None, 0, None) == -3


def test_workspace_sizes_grow_with_the_problem(L):
    a = L.provip_head_scores_workspace_size(8, 1091, 8, 96, 960, 2, 1)
    b = L.provip_head_scores_workspace_size(16, 1091, 8, 96, 960, 2, 1)
    assert 0 < a < b
    assert L.provip_prune_workspace_size(8, 1091, 8, 96, 960, 2, 1) == a
    assert L.provip_similarity_reduce_workspace_size(1, 9216, 3584, 128, 2304) > \
        L.provip_relevance_workspace_size(1, 9216, 3584, 128)


def test_schedule_rejects_inconsistent_stages():
    """The progressive schedule validates its stage arguments before touching
    the GPU."""
    from paper_2608_25332_gb300.schedule import ProgressiveSchedule
    with pytest.raises(ValueError):  # without pre-LLM pruning every visual token reaches the LLM
        ProgressiveSchedule(2, 576, 4096, 128, 739, 32, 32, 4096, 1, 288, 73, 20, 6, pre_llm=False)
    with pytest.raises(ValueError):
        ProgressiveSchedule(2, 576, 4096, 128, 739, 32, 32, 4096, 1, 576, 73, 20, 6, shallow_heads="some")


def test_missing_library_fails_loudly(tmp_path, monkeypatch):
    """No fallback: with the compiled library absent, the first call raises."""
    from paper_2608_25332_gb300 import provip
    monkeypatch.setattr(provip, "_lib", None)
    monkeypatch.setattr(provip, "LIB_PATH", str(tmp_path / "libprovip.so"))
    with pytest.raises(provip.ProvipError, match="not built"):
        provip.lib()
