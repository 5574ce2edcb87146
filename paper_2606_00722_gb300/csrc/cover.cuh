// Regular-cover group test (Sec. 4.3, Alg. 4's RelaxedSelect): L(F_G) cap L(A_x) != empty
// by forward state-set simulation of the flattened recursive transition
// network F_G over the partial-output graph.
//
// F_G's states are the dotted items (p, d) -- numbered exactly like the
// Earley items, so a terminal transition (p, d) -a-> (p, d+1) is the same
// ((set & EXP_T[a]) << 1) -- followed by entry(A) = D + A and exit(A) =
// D + V + A.  Epsilon edges: entry(A) -> (p, 0) for every p with lhs A;
// (p, d) -> entry(B) when B follows the dot; (p, |rhs|) -> exit(lhs p);
// exit(B) -> (p, d+1) at every occurrence of B.  Every call site shares the
// one entry(B), which is what forgets the return site.  A node's set is
// closed under epsilon edges (under every edge at a gap, the Sigma_lex*
// self-loop), using closure rows precomputed per state on the host.
#pragma once
#include "walk.cuh"

namespace epic {

constexpr int kMaxFW = 512;

class CoverCols {
 public:
  static constexpr bool kRecord = false;
  const DevGrammar& g;
  Workspace ws;
  WsDims dims;
  WalkShared& sh;
  int W, FW;
  __device__ CoverCols(const DevGrammar& g_, Workspace w, WsDims d, WalkShared& shared)
      : g(g_), ws(w), dims(d), sh(shared), W(g_.W), FW(g_.FW) {}

  __device__ void reset() {
    if (threadIdx.x == 0) {
      sh.ncols = 0;
      sh.status = kWalkOk;
    }
    __syncthreads();
  }
  __device__ void cleanup() {}
  __device__ int open_column() {
    int c = sh.ncols;
    if (c >= dims.nmax || c >= kMaxCols) {
      if (threadIdx.x == 0) sh.status = kWalkOverflow;
      return -1;
    }
    for (int w = threadIdx.x; w < FW; w += blockDim.x) ws.cov[(size_t)c * FW + w] = 0;
    if (threadIdx.x == 0) sh.scratch_i[0] = c;
    __syncthreads();
    return c;
  }
  __device__ void seed(int c) {
    if (threadIdx.x == 0) ws.cov[(size_t)c * FW + (g.cov_start >> 5)] |= 1u << (g.cov_start & 31);
    __syncthreads();
  }
  // dst |= src (epsilon) or dst |= shift(src & lbl) over the item words
  __device__ void arrive_labels(int src, bool eps) {
    int c = sh.scratch_i[0];
    const uint32_t* s = ws.cov + (size_t)src * FW;
    uint32_t* d = ws.cov + (size_t)c * FW;
    if (eps) {
      for (int w = threadIdx.x; w < FW; w += blockDim.x) d[w] |= s[w];
    } else {
      for (int w = threadIdx.x; w < W; w += blockDim.x) {
        uint32_t v = s[w] & sh.lbl[w];
        uint32_t p = w > 0 ? (s[w - 1] & sh.lbl[w - 1]) : 0u;
        d[w] |= (v << 1) | (p >> 31);
      }
    }
    __syncthreads();
  }
  __device__ void close_column(int c, bool gap) {
    __shared__ uint32_t R[kMaxFW];
    const uint32_t* rows = gap ? g.cov_all_close : g.cov_eps_close;
    uint32_t* S = ws.cov + (size_t)c * FW;
    for (int w = threadIdx.x; w < FW; w += blockDim.x) R[w] = 0;
    __syncthreads();
    int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nwarps = blockDim.x >> 5;
    // each warp takes every nwarps-th set state and ORs its closure row
    int seen = 0;
    for (int w = 0; w < FW; ++w) {
      uint32_t m = S[w];
      while (m) {
        int b = __ffs(m) - 1;
        m &= m - 1;
        if ((seen++ % nwarps) != warp) continue;
        const uint32_t* r = rows + (size_t)((w << 5) + b) * FW;
        for (int v = lane; v < FW; v += 32)
          if (r[v]) atomicOr(&R[v], r[v]);
      }
    }
    __syncthreads();
    for (int w = threadIdx.x; w < FW; w += blockDim.x) S[w] = R[w];
    __syncthreads();
  }
  __device__ void finish_column(int c) {
    __shared__ int nz;
    if (threadIdx.x == 0) nz = 0;
    __syncthreads();
    for (int w = threadIdx.x; w < FW; w += blockDim.x)
      if (ws.cov[(size_t)c * FW + w]) nz = 1;
    __syncthreads();
    if (threadIdx.x == 0) {
      ws.col_off[c] = nz;
      sh.ncols = c + 1;
    }
    __syncthreads();
  }
  __device__ bool column_empty(int c) const { return ws.col_off[c] == 0; }
  __device__ bool column_has_accept(int c, int /*start*/) {
    return (ws.cov[(size_t)c * FW + (g.cov_accept >> 5)] >> (g.cov_accept & 31)) & 1u;
  }
};

}  // namespace epic
