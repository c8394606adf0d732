"""The C ABI used from a plain C++ host program, with no Python or PyTorch in
the process: the program includes only include/acid.h and the CUDA runtime
API, links libacid_gb300.so, and checks closed forms.

* drift: prev_i = 1 + (i mod 7), cur_i = 1.25 prev_i over 1,000,003 fp32
  elements (a ragged count) gives rel_l1 = 0.25 exactly (every term and
  partial sum is exactly representable), through a host output pointer;
* cache apply: out = x + r element for element;
* the zero-denominator reading: rel_l1(0, 0) = 0 and rel_l1(0, c != 0) = inf.
"""

import os
import shutil
import subprocess

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2607_12358_gb300")

SOURCE = r"""
#include <cmath>
#include <cstdio>
#include <vector>
#include <cuda_runtime.h>
#include "acid.h"

#define CHECK(x) do { acid_status st = (x); if (st != ACID_OK) { \
  std::printf("FAIL %s: %d %s\n", #x, (int)st, acid_last_error()); return 1; } } while (0)

static double drift(const std::vector<float>& prev, const std::vector<float>& cur) {
  const int64_t n = (int64_t)prev.size();
  float *dp = nullptr, *dc = nullptr;
  void* ws = nullptr;
  size_t wsb = 0;
  if (acid_drift_workspace_size(n, &wsb) != ACID_OK) return -1.0;
  if (cudaMalloc(&dp, n * sizeof(float)) || cudaMalloc(&dc, n * sizeof(float)) || cudaMalloc(&ws, wsb)) return -2.0;
  cudaMemcpy(dp, prev.data(), n * sizeof(float), cudaMemcpyHostToDevice);
  cudaMemcpy(dc, cur.data(), n * sizeof(float), cudaMemcpyHostToDevice);
  double rel = -3.0;  // host pointer: the call returns with the value written
  if (acid_drift_signal(dp, dc, n, ACID_FP32, &rel, nullptr, ws, wsb, nullptr) != ACID_OK) rel = -4.0;
  cudaFree(dp);
  cudaFree(dc);
  cudaFree(ws);
  return rel;
}

int main() {
  const int64_t n = 1000003;
  std::vector<float> prev(n), cur(n), r(n), out(n);
  for (int64_t i = 0; i < n; ++i) {
    prev[i] = 1.0f + (float)(i % 7);
    cur[i] = 1.25f * prev[i];
    r[i] = 0.5f * (float)(i % 5) - 1.0f;
  }
  const double rel = drift(prev, cur);
  std::printf("rel_l1 %.17g\n", rel);
  if (rel != 0.25) { std::printf("FAIL drift\n"); return 1; }

  std::vector<float> z(1000, 0.0f), c(1000, 2.0f);
  const double zz = drift(z, z), zc = drift(z, c);
  std::printf("zero %.17g inf %.17g\n", zz, zc);
  if (zz != 0.0 || !std::isinf(zc)) { std::printf("FAIL zero denominator\n"); return 1; }

  float *dx = nullptr, *dr = nullptr, *dout = nullptr;
  if (cudaMalloc(&dx, n * 4) || cudaMalloc(&dr, n * 4) || cudaMalloc(&dout, n * 4)) return 1;
  cudaMemcpy(dx, cur.data(), n * 4, cudaMemcpyHostToDevice);
  cudaMemcpy(dr, r.data(), n * 4, cudaMemcpyHostToDevice);
  CHECK(acid_cache_apply(dx, dr, dout, n, ACID_FP32, nullptr));
  cudaMemcpy(out.data(), dout, n * 4, cudaMemcpyDeviceToHost);
  for (int64_t i = 0; i < n; ++i)
    if (out[i] != cur[i] + r[i]) { std::printf("FAIL cache apply at %lld\n", (long long)i); return 1; }
  CHECK(acid_check_device_error());
  std::printf("launches %lld\n", (long long)acid_launch_count());
  std::printf("OK\n");
  return 0;
}
"""


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__ as g

    g.build()
    path = os.path.join(PKG, "libacid_gb300.so")
    assert os.path.exists(path)
    return path


def test_c_program_against_closed_forms(lib, tmp_path):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    src = tmp_path / "acid_c_client.cu"
    src.write_text(SOURCE)
    exe = tmp_path / "acid_c_client"
    subprocess.run([nvcc, "-O2", "-std=c++17", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe),
                    "-L", PKG, "-lacid_gb300", "-Xlinker", "-rpath=" + PKG], check=True, capture_output=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0 and "OK" in r.stdout, r.stdout + r.stderr
    assert "rel_l1 0.25" in r.stdout
