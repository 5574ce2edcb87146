// Measurement entry point: the integer-pipe peak of this GPU for the word
// operations the bit-parallel Earley sweeps issue (logic on 32-bit words and
// funnel shifts), used as the denominator of the walks' roofline.  Not part
// of the method (see include/epic_measure.h).
#include <cuda_runtime.h>

#include <cstdint>

#include "../../include/epic_measure.h"

namespace {

// Every thread runs kChains independent chains; each iteration is one LOP3
// (three-input logic: the and/or/xor of the sweeps) and one SHF (funnel shift:
// the one-bit item advance across words) per chain, 2 word operations.
constexpr int kChains = 8;
constexpr int kIters = 4096;

__global__ void k_int_peak(uint32_t* out, uint32_t seed) {
  uint32_t a[kChains], b[kChains];
#pragma unroll
  for (int c = 0; c < kChains; ++c) {
    a[c] = seed * (threadIdx.x + 1 + c) + blockIdx.x;
    b[c] = seed ^ (c * 0x9E3779B9u + threadIdx.x);
  }
  for (int it = 0; it < kIters; ++it) {
#pragma unroll
    for (int c = 0; c < kChains; ++c) {
      uint32_t r;
      asm volatile("lop3.b32 %0, %1, %2, %3, 0xE8;" : "=r"(r) : "r"(a[c]), "r"(b[c]), "r"(a[(c + 1) % kChains]));
      uint32_t s;
      asm volatile("shf.l.wrap.b32 %0, %1, %2, 1;" : "=r"(s) : "r"(r), "r"(b[c]));
      a[c] = r;
      b[c] = s;
    }
  }
  uint32_t acc = 0;
#pragma unroll
  for (int c = 0; c < kChains; ++c) acc ^= a[c] ^ b[c];
  if (acc == 0x12345678u) out[0] = acc;  // keeps the chains live
}

}  // namespace

extern "C" int epic_measure_int_peak(double* word_ops_per_s, double* ms, void* cuda_stream) {
  if (!word_ops_per_s) return 1;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return 5;
  uint32_t* out = nullptr;
  if (cudaMalloc(&out, 4) != cudaSuccess) return 4;
  const int threads = 512, blocks = sms * 4;  // 2048 threads per SM: full occupancy
  cudaEvent_t e0, e1;
  cudaEventCreate(&e0);
  cudaEventCreate(&e1);
  float best = 1e30f;
  for (int rep = 0; rep < 4; ++rep) {  // the first is a warm-up
    cudaEventRecord(e0, st);
    k_int_peak<<<blocks, threads, 0, st>>>(out, 0x2545F491u + rep);
    cudaEventRecord(e1, st);
    cudaEventSynchronize(e1);
    float t = 0.f;
    cudaEventElapsedTime(&t, e0, e1);
    if (rep > 0 && t < best) best = t;
  }
  const bool ok = cudaGetLastError() == cudaSuccess;
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  cudaFree(out);
  if (!ok) return 5;
  const double ops = (double)blocks * threads * kIters * kChains * 2.0;
  *word_ops_per_s = ops / (best * 1e-3);
  if (ms) *ms = best;
  return 0;
}
