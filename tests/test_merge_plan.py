"""Host logic of the merge Gram on pairs of SMs (Sec. 4.3, nearest kept token):
the tile plan and its deal, compiled from the library's own source into a small
host program (no GPU), checked on the workloads' shapes and on ragged and
seeded random ones: every pruned row gets each partial slot exactly once, every
column range is 1..256 wide with a planned box height, and every tile is dealt
to exactly one pair."""
import os
import shutil
import subprocess

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))


def _nvcc():
    for c in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if c and os.path.exists(c):
            return c
    return None


@pytest.fixture(scope="module")
def checker(tmp_path_factory):
    cc = _nvcc()
    if cc is None:
        pytest.skip("nvcc not found")
    out = str(tmp_path_factory.mktemp("plan") / "merge_plan_check")
    root = os.path.dirname(HERE)
    r = subprocess.run([cc, "-std=c++17", "-O1", "-gencode", "arch=compute_103a,code=sm_103a",
                        "-I" + os.path.join(root, "include"), os.path.join(HERE, "merge_plan_check.cu"),
                        "-o", out], capture_output=True, text=True)
    assert r.returncode == 0, r.stdout + r.stderr
    return out


def _run(checker, shapes):
    args = [str(v) for s in shapes for v in s]
    r = subprocess.run([checker, *args], capture_output=True, text=True)
    assert r.returncode == 0, r.stdout + r.stderr
    lines = r.stdout.splitlines()
    assert len(lines) == len(shapes), r.stdout
    for (B, N_v, keep, D, sms), line in zip(shapes, lines):
        # a plan exists whenever 16 ranges rounded to 32 columns stay within
        # 256 (keep <= 16 * 224); above that the single-SM form may take over
        assert line.startswith("ok ") or (line.startswith("noplan") and keep > 16 * 224), line


def test_plans_of_the_workloads_and_ragged_shapes(checker):
    # (B, N_v, keep, D, SMs)
    _run(checker, [
        (8, 2880, 960, 4096, 152), (1, 9216, 2304, 3584, 152), (16, 576, 288, 4096, 152),
        (32, 576, 192, 5120, 152), (6, 1000, 237, 256, 152), (2, 700, 640, 136, 152),
        (5, 513, 1, 128, 152), (3, 800, 130, 64, 152), (40, 800, 500, 64, 152), (3, 37, 1, 64, 152),
        (3, 37, 36, 64, 152), (64, 2880, 960, 4096, 152), (8, 2880, 960, 4096, 132), (1, 600, 1, 64, 2),
    ])


def test_plans_of_random_shapes(checker):
    rng = np.random.default_rng(20260)
    shapes = []
    for _ in range(60):
        N_v = int(rng.integers(2, 6000))
        keep = int(rng.integers(1, min(N_v - 1, 4096) + 1))
        shapes.append((int(rng.integers(1, 24)), N_v, keep, 8 * int(rng.integers(1, 600)),
                       2 * int(rng.integers(1, 90))))
    _run(checker, shapes)
