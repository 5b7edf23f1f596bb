"""The attention kernel's weights come from ex2.approx.ftz.f32 (2^t on the
special-function unit), and its tolerance counts that instruction's error
as at most 2 ulp (2^-22 relative).  This measures it on the GPU against
exp2 in fp64 over every fp32 t in [-126, 0] (the range the kernel feeds it:
arguments above 0 stay below 8 and are scaled into it by the reference
maximum's definition, so the range checked is the part where relative
accuracy matters).  A tiny standalone program, compiled with nvcc."""
import os
import shutil
import subprocess

import pytest

pytestmark = pytest.mark.gpu

NVCC = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"

SRC = r"""
#include <cstdio>
#include <cstdint>
#include <cstring>
#include <cmath>
#include <cuda_runtime.h>
__global__ void k(uint32_t lo, uint32_t n, unsigned long long* worst) {
  const uint32_t stride = gridDim.x * blockDim.x;
  double w = 0.0;
  for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    const float x = __uint_as_float(lo + i);
    if (!(x >= -126.0f && x <= 0.0f)) continue;
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    const double r = exp2((double)x);
    const double e = fabs((double)y - r) / r;
    w = e > w ? e : w;
  }
  atomicMax(worst, (unsigned long long)__double_as_longlong(w));  // w >= 0: its bits order like its value
}
int main() {
  unsigned long long* d;
  if (cudaMalloc(&d, 8) != cudaSuccess) return 2;
  cudaMemset(d, 0, 8);
  const uint32_t lo = 0x80000000u, hi = 0xC2FC0000u;  // -0 .. -126
  k<<<1216, 256>>>(lo, hi - lo + 1u, d);
  if (cudaDeviceSynchronize() != cudaSuccess) return 3;
  unsigned long long h = 0;
  cudaMemcpy(&h, d, 8, cudaMemcpyDeviceToHost);
  double w;
  memcpy(&w, &h, 8);
  printf("%.6e\n", w);
  return 0;
}
"""


@pytest.mark.skipif(not os.path.exists(NVCC), reason="nvcc not found")
def test_ex2_approx_within_two_ulp(tmp_path):
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    src = tmp_path / "ex2.cu"
    src.write_text(SRC)
    exe = tmp_path / "ex2"
    r = subprocess.run([NVCC, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-o", str(exe), str(src)],
                       capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    worst = float(r.stdout.strip())
    assert 0.0 < worst <= 2.0 ** -22, worst
