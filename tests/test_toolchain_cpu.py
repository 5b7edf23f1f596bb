"""What the CUDA 13 toolchain accepts for sm_103a (GB300), checked by
compiling: the int8 kind of the fifth-generation tensor-core MMA
(tcgen05.mma ... kind::i8) is refused, while the 16-bit kind assembles.
This is why the layer's int8 dot-4 (Algorithm 1's vpdpbusd) runs on dp4a
and why a tensor-core route would have to carry int8 values as f16/bf16.
Only ptxas's message is read; nothing compiled is inspected."""
import os
import shutil
import subprocess

import pytest

NVCC = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"

SRC = r"""
__global__ void k(unsigned long long adesc, unsigned long long bdesc, unsigned idesc, unsigned tmem) {
    asm volatile("{\n .reg .pred p;\n setp.ne.u32 p, %3, 0;\n"
                 " tcgen05.mma.cta_group::1.kind::KIND [%0], %1, %2, %3, p;\n}\n"
                 :: "r"(tmem), "l"(adesc), "l"(bdesc), "r"(idesc));
}
"""


def _compile(tmp_path, kind: str):
    src = tmp_path / f"mma_{kind}.cu"
    src.write_text(SRC.replace("KIND", kind))
    return subprocess.run([NVCC, "-gencode", "arch=compute_103a,code=sm_103a", "-c", str(src), "-o",
                           str(tmp_path / f"mma_{kind}.o")], capture_output=True, text=True, timeout=120)


@pytest.mark.skipif(not os.path.exists(NVCC), reason="nvcc not found")
def test_tcgen05_kind_i8_is_refused_for_sm_103a(tmp_path):
    r = _compile(tmp_path, "i8")
    assert r.returncode != 0
    assert "kind::i8" in r.stderr and "sm_103a" in r.stderr


@pytest.mark.skipif(not os.path.exists(NVCC), reason="nvcc not found")
def test_tcgen05_kind_f16_assembles_for_sm_103a(tmp_path):
    r = _compile(tmp_path, "f16")
    assert r.returncode == 0, r.stderr
