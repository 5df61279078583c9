"""bench.py's host-side helpers (no GPU): the launch count per call that gpu_launches is built
from, and the code hash that keeps a recorded DRAM traffic figure tied to the kernel it was
measured on."""
import os
import shutil
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2608_18656_gb300 import inputs as I  # noqa: E402


class FakeFav:
    PATH_SIMT, PATH_DECODE, PATH_PREFILL = 1, 2, 3

    def __init__(self, path, splits=0):
        self.path, self.splits = path, splits

    def last_path(self):
        return self.path

    def last_decode_splits(self):
        return self.splits


@pytest.mark.parametrize("path,splits,dtype,expected", [
    (3, 0, I.F16, 1),      # fp16 prefill: the prefill kernel only
    (3, 0, I.BF16, 3),     # bf16 prefill: V max, V to fp16, prefill
    (2, 1, I.F16, 1),      # decode with one split writes O directly
    (2, 8, I.BF16, 2),     # decode with splits: + the split merge
    (1, 0, I.F32, 1),      # CUDA-core kernel
])
def test_launches_per_call(path, splits, dtype, expected):
    w = I.Workload("t", dtype, 1, 2, 2, 8, 8, 64, False, False, 0)
    assert bench.launches_per_call(FakeFav(path, splits), w) == expected


def test_kernel_hash_ignores_comments_but_not_code(tmp_path, monkeypatch):
    src = os.path.join(ROOT, "paper_2608_18656_gb300", "csrc")
    root = tmp_path / "repo"
    shutil.copytree(src, root / "paper_2608_18656_gb300" / "csrc")
    monkeypatch.setattr(bench, "ROOT", str(root))
    h0 = bench.kernel_hash()
    f = root / "paper_2608_18656_gb300" / "csrc" / "fav_prefill.cu"
    text = f.read_text()
    f.write_text("// a new comment line\n/* and a block\n   comment */\n" + text + "\n\n")
    assert bench.kernel_hash() == h0
    changed = text.replace("kRescaleThreshold = 4.0f", "kRescaleThreshold = 3.0f", 1)
    assert changed != text                  # the constant this test edits still exists
    f.write_text(changed)
    assert bench.kernel_hash() != h0
