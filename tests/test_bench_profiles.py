"""The bench reports a kernel's DRAM traffic from a committed ncu summary only
while that summary was taken on the kernel's current code.  A summary names
the sha256[:16] of the .cu file or of its code alone (comments and blank
space removed), so that comment-only edits keep a capture valid while any
change to the code drops it (host only, no GPU)."""
import hashlib
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
bench = pytest.importorskip("bench")

SRC = b"""// a kernel
__global__ void k(float *y) {  /* one store */
    y[0] = 1.0f;   // the value
}
"""


def test_code_sha_ignores_comments_and_layout():
    relaid = b"""/* another header,
   two lines */
__global__ void k(float *y)
{
    y[0] = 1.0f;
}
"""
    assert bench.code_sha(SRC) == bench.code_sha(relaid)
    assert bench.code_sha(SRC) != hashlib.sha256(SRC).hexdigest()[:16]


def test_code_sha_sees_code_changes():
    for changed in (SRC.replace(b"1.0f", b"2.0f"), SRC.replace(b"y[0]", b"y[1]"),
                    SRC.replace(b"float *y", b"double *y")):
        assert bench.code_sha(changed) != bench.code_sha(SRC)


def test_traffic_lines_of_the_decode_profile_match_the_kernels():
    """The 70B decode summary's traffic lines name the current code of both
    decode kernels (re-capture after a code change, then update them)."""
    for kernel in ("decode_tc.cu", "gemv_decode.cu"):
        t = bench.profile_traffic(kernel, "gemm_decode_llama2_70b_decode.md")
        assert t is not None and t > 3e8, kernel


def test_a_stale_sha_reports_no_traffic(tmp_path, monkeypatch):
    prof = tmp_path / "profiles"
    csrc = tmp_path / "paper_2607_17733_gb300" / "csrc"
    prof.mkdir()
    csrc.mkdir(parents=True)
    (csrc / "k.cu").write_bytes(SRC)
    (prof / "k.md").write_text("traffic_bytes_per_launch: 1000 kernel_sha: 0123456789abcdef\n"
                               f"traffic_bytes_per_launch: 2000 kernel_sha: {bench.code_sha(SRC)}\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.profile_traffic("k.cu", "k.md") == 2000.0
    (csrc / "k.cu").write_bytes(SRC.replace(b"1.0f", b"3.0f"))
    assert bench.profile_traffic("k.cu", "k.md") is None
