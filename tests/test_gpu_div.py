"""The encoder's fp64 division on the integer pipes (div_recip / div_rn in
csrc/seedq_internal.cuh) against the GPU's IEEE division, bit for bit.

div_rn must return the correctly rounded quotient for every operand pair the
encoder can produce (and falls back to the hardware division outside its
range), so the check runs it on random operands over a wide exponent range and
on edge operands: significands at 1 and just below 2, quotients whose exponent
sits at either end of the normal range, zero numerators, both signs, and
quotients that fall exactly on representable values.
"""
import os
import shutil
import subprocess

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2609_38477_gb300", "csrc")

pytestmark = pytest.mark.gpu

SOURCE = r"""
#include <cstdio>
#include <cstdlib>
#include <cstdint>
#include <vector>
#include "seedq_internal.cuh"

__global__ void k_div(const double *a, const double *b, int64_t n, unsigned long long *bad,
                      double *first) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const seedq::DivRecip r = seedq::div_recip(b[i]);
    const double q = seedq::div_rn(a[i], r);
    const double h = __ddiv_rn(a[i], b[i]);
    if (__double_as_longlong(q) != __double_as_longlong(h)) {
      const unsigned long long k = atomicAdd(bad, 1ull);
      if (k == 0) { first[0] = a[i]; first[1] = b[i]; first[2] = q; first[3] = h; }
    }
  }
}

int main(int argc, char **argv) {
  FILE *f = fopen(argv[1], "rb");
  int64_t n = 0;
  if (!f || fread(&n, 8, 1, f) != 1) return 2;
  std::vector<double> a(n), b(n);
  if (fread(a.data(), 8, n, f) != (size_t)n || fread(b.data(), 8, n, f) != (size_t)n) return 2;
  fclose(f);
  double *da, *db, *dfirst;
  unsigned long long *dbad;
  cudaMalloc(&da, 8 * n);
  cudaMalloc(&db, 8 * n);
  cudaMalloc(&dbad, 8);
  cudaMalloc(&dfirst, 32);
  cudaMemcpy(da, a.data(), 8 * n, cudaMemcpyHostToDevice);
  cudaMemcpy(db, b.data(), 8 * n, cudaMemcpyHostToDevice);
  cudaMemset(dbad, 0, 8);
  k_div<<<1024, 256>>>(da, db, n, dbad, dfirst);
  unsigned long long bad = 0;
  double first[4] = {0, 0, 0, 0};
  cudaMemcpy(&bad, dbad, 8, cudaMemcpyDeviceToHost);
  cudaMemcpy(first, dfirst, 32, cudaMemcpyDeviceToHost);
  const cudaError_t e = cudaDeviceSynchronize();
  printf("%s %lld %llu %.17g %.17g %.17g %.17g\n", cudaGetErrorName(e), (long long)n, bad, first[0], first[1],
         first[2], first[3]);
  return e == cudaSuccess ? 0 : 1;
}
"""


def _operands(n_random: int) -> tuple[np.ndarray, np.ndarray]:
    rng = np.random.default_rng(7)
    # random significands and exponents (both signs), quotients across the range
    a = rng.uniform(1, 2, n_random) * np.exp2(rng.integers(-600, 600, n_random).astype(np.float64))
    b = rng.uniform(1, 2, n_random) * np.exp2(rng.integers(-400, 400, n_random).astype(np.float64))
    a *= np.where(rng.random(n_random) < 0.5, -1.0, 1.0)
    b *= np.where(rng.random(n_random) < 0.5, -1.0, 1.0)
    sig = np.array([1.0, np.nextafter(1.0, 2.0), np.nextafter(2.0, 1.0), 1.5, 1.25, np.nextafter(1.5, 1.0)])
    ea, eb = np.meshgrid(sig, sig)
    ea, eb = ea.ravel(), eb.ravel()
    edge_a, edge_b = [], []
    # significand edges at ordinary exponents
    for sa in (1, -1):
        edge_a.append(sa * ea * 8.0)
        edge_b.append(eb * 0.25)
    # quotient exponents at and around the ends of the normal range (the fast
    # path covers -1021..1022 and hands the rest to the hardware division):
    # a = ea 2^ka, b = eb 2^kb with ka - kb = eq, both operands normal
    for eq in list(range(-1030, -1014)) + list(range(1014, 1024)):
        ka, kb = (eq, 0) if eq > 0 else (-500, -500 - eq)
        edge_a.append(ea * np.exp2(float(ka)))
        edge_b.append(eb * np.exp2(float(kb)))
        edge_a.append(-ea * np.exp2(float(ka)))
        edge_b.append(eb * np.exp2(float(kb)))
    # exact quotients (small integers) and zero numerators
    ints = np.arange(1, 2000, dtype=np.float64)
    edge_a.append(ints * 3.0)
    edge_b.append(np.full(ints.size, 3.0))
    edge_a.append(np.zeros(50))
    edge_b.append(rng.uniform(1, 2, 50))
    edge_a.append(-np.zeros(50))
    edge_b.append(-rng.uniform(1, 2, 50))
    ae = np.concatenate(edge_a)
    be = np.concatenate(edge_b)
    keep = np.isfinite(ae) & np.isfinite(be) & (be != 0)
    return np.concatenate([a, ae[keep]]), np.concatenate([b, be[keep]])


@pytest.mark.skipif(shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"),
                    reason="needs nvcc")
def test_div_rn_matches_hardware_division(tmp_path):
    import torch

    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    nvcc = "/usr/local/cuda/bin/nvcc" if os.path.exists("/usr/local/cuda/bin/nvcc") else "nvcc"
    src = tmp_path / "div.cu"
    src.write_text(SOURCE)
    exe = tmp_path / "div"
    r = subprocess.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17", "-I", CSRC,
                        str(src), "-o", str(exe)], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr[-3000:]
    a, b = _operands(1 << 22)
    data = tmp_path / "ops.bin"
    with open(data, "wb") as f:
        f.write(np.int64(a.size).tobytes())
        f.write(a.astype(np.float64).tobytes())
        f.write(b.astype(np.float64).tobytes())
    r = subprocess.run([str(exe), str(data)], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    status, n, bad, *first = r.stdout.split()
    assert status == "cudaSuccess", r.stdout
    assert int(n) == a.size and int(bad) == 0, r.stdout
