// Workspace layouts shared by the host side and the kernels: the per-CTA
// block-walk workspace (WsPack), the per-warp walk workspace (WPack), the
// shared-memory staging sizes, and the statistics slots.
#pragma once
#include "skeleton.cuh"
#include "warpwalk.cuh"

namespace epic {

constexpr int kMaxSel = 64;  // proposed positions per sequence that selection handles

struct WsPack {
  char* base;
  size_t per_cta;
  WsDims dims;
  int W, VW, FW;
  __device__ void carve(int cta, Workspace& ws, WalkScratch& sc) const {
    char* p = base + per_cta * (size_t)cta;
    auto take = [&](size_t bytes) {
      char* r = p;
      p += (bytes + 255) & ~(size_t)255;
      return r;
    };
    int nm = dims.nmax;
    ws.stage = (uint32_t*)take((size_t)nm * W * 4);
    ws.bdone = (uint32_t*)take((size_t)nm * VW * 4);
    ws.col_off = (int32_t*)take((size_t)(nm + 1) * 4);
    ws.cov = (uint32_t*)take((size_t)nm * FW * 4);
    sc.g_src = (int32_t*)take(kMaxQ * 4);
    sc.g_end = (int32_t*)take(kMaxQ * 4);
    sc.g_len = (int32_t*)take(kMaxQ * 4);
    sc.g_last = (int32_t*)take(kMaxQ * 4);
    sc.f_q = (int32_t*)take(kMaxQ * 4);
    sc.f_c = (int32_t*)take(kMaxQ * 4);
    sc.key_q = (int32_t*)take(kMaxQ * 4);
    sc.g_tail = (uint8_t*)take(kMaxQ * 16);
    sc.g_lbl = (uint32_t*)take(kMaxQ * 8 * 4);
    sc.expn = (uint32_t*)take((size_t)nm * W * 4);
    sc.bnew = (uint32_t*)take((size_t)nm * VW * 4);
    ws.org = (int32_t*)take((size_t)dims.emax * 4);
    ws.bits = (uint32_t*)take((size_t)dims.emax * W * 4);
  }
};

inline size_t ws_bytes_per_cta(const WsDims& d, int W, int VW, int FW) {
  auto r = [](size_t b) { return (b + 255) & ~(size_t)255; };
  size_t nm = d.nmax;
  return r(nm * W * 4) + r(nm * VW * 4) + r((nm + 1) * 4) + r(nm * FW * 4) + 7 * r(kMaxQ * 4) +
         r(kMaxQ * 16) + r(kMaxQ * 32) + r(nm * W * 4) + r(nm * VW * 4) + r((size_t)d.emax * 4) +
         r((size_t)d.emax * W * 4);
}

enum StatIdx {
  S_CHECKS, S_VALID, S_OVERFLOW, S_BAD, S_COLUMNS, S_ENTRIES, S_COVER, S_EXACT, S_SELECTED,
  S_FB_CHECKS, S_FB_COMMITS, S_LEX_LOOKUPS, S_LEX_MISSES, S_LEX_UNCACHED, S_WITNESS_FAIL, S_N
};
constexpr int kMaxFallbackCand = 4096;  // proposed (position, candidate) pairs per sequence of the fallback
constexpr int kMaxFallbackSpec = 16;    // fallback tests of one sequence in one round

// shared-memory staging of one warp: rows, completed-NT sets, slot origins,
// origin slots (16-byte multiple)
__host__ __device__ inline size_t smem_per_warp(int nmax, int rmax, int W, int VW) {
  size_t b = (size_t)rmax * W * 4 + (size_t)rmax * VW * 4 + (size_t)rmax * 4 + (size_t)rmax * 8 + (size_t)nmax * 2;
  return (b + 15) & ~(size_t)15;
}

struct WPack {
  char* base;
  size_t per_warp;
  int nmax;
  long long emax;
  int W, VW;
  __device__ WWs carve(long long warp) const {
    WWs ws;
    char* p = base + per_warp * (size_t)warp;
    auto take = [&](size_t bytes) {
      char* r = p;
      p += (bytes + 255) & ~(size_t)255;
      return r;
    };
    ws.stage = (uint32_t*)take((size_t)nmax * W * 4);
    ws.bdone = (uint32_t*)take((size_t)nmax * VW * 4);
    ws.col_off = (int32_t*)take((size_t)(nmax + 1) * 4);
    ws.f_q = (int32_t*)take(kWMaxQ * 4);
    ws.f_c = (int32_t*)take(kWMaxQ * 4);
    ws.g_src = (int32_t*)take(kWMaxQ * 4);
    ws.g_end = (int32_t*)take(kWMaxQ * 4);
    ws.g_len = (int32_t*)take(kWMaxQ * 4);
    ws.g_last = (int32_t*)take(kWMaxQ * 4);
    ws.key_q = (int32_t*)take(kWMaxQ * 4);
    ws.g_tail = (uint32_t*)take(kWMaxQ * 16);
    ws.g_lbl = (uint32_t*)take(kWMaxQ * 32);
    ws.ssum = (uint32_t*)take((size_t)nmax * 8);
    ws.org = (int32_t*)take((size_t)emax * 4);
    ws.esum = (uint32_t*)take((size_t)emax * 8);
    ws.bits = (uint32_t*)take((size_t)emax * W * 4);
    return ws;
  }
};

inline size_t wbytes_per_warp(int nmax, long long emax, int W, int VW) {
  auto r = [](size_t b) { return (b + 255) & ~(size_t)255; };
  return r((size_t)nmax * W * 4) + r((size_t)nmax * VW * 4) + r((size_t)(nmax + 1) * 4) + 7 * r(kWMaxQ * 4) +
         r(kWMaxQ * 16) + r(kWMaxQ * 32) + r((size_t)nmax * 8) + r((size_t)emax * 4) + r((size_t)emax * 8) +
         r((size_t)emax * W * 4);
}

// Bytes of the grammar tables the warp walk reads, staged in shared memory
// (16-byte aligned pieces).
__host__ __device__ inline size_t gtab_bytes(int T, int V, int W, int D, int Q) {
  auto r = [](size_t b) { return (b + 15) & ~(size_t)15; };
  return r((size_t)T * W * 4) + 2 * r((size_t)V * W * 4) + r((size_t)V * W * 4) + 5 * r((size_t)W * 4) +
         2 * r((size_t)D * 2) + r((size_t)Q * 2) + r((size_t)Q) + r((size_t)T);
}

}  // namespace epic
