// Alg. 4 (relaxed compatible-subset selection with exact re-check): kernels
// and launchers.
#include <cuda_runtime.h>

#include "launch.h"

using namespace epic;

// Selection and the fallback run one CTA per walk: 16 warps share each
// column closure (the Gauss-Seidel engine's width, as the forward charts).
constexpr int kSelThreads = 32 * kGsMaxWarps;

// Alg. 4 per sequence: one CTA runs RelaxedSelect / ExactShrink with an
// explicit stack; thread 0 drives the recursion, the whole CTA runs each
// cover test (CoverCols walk) and exact joint check (a walk with the
// Gauss-Seidel columns of gscols.cuh, the grammar's per-item tables staged in
// dynamic shared memory).

struct SelFrame {
  int8_t kind;  // 0 root, 1 relaxed, 2 shrink
  int8_t pc;
  unsigned long long base, set, a, b;
};

// Alg. 4 always starts with the cover test of x (+) C and, when that passes,
// continues with the exact test of the same x (+) C.  Both are run here at
// once, one CTA each per sequence, before the recursion; k_select reuses the
// two answers when it asks for exactly these tests.  spec[b] = {cover,
// exact}: 1 pass, 0 fail, -1 not available (overflow / bad input).
__global__ void __launch_bounds__(kSelThreads) k_select_spec(DevGrammar g, const LexEntry* __restrict__ table, int vocab,
                                                          const int32_t* __restrict__ x, int B, int n,
                                                          const int32_t* __restrict__ pos, int k,
                                                          const int32_t* __restrict__ tok, int8_t* __restrict__ spec,
                                                          WsPack wsp) {
  __shared__ WalkShared sh;
  __shared__ GsShared gss;
  __shared__ int s_pos[kMaxSel], s_tok[kMaxSel];
  __shared__ int ns;
  extern __shared__ __align__(16) unsigned char dyn[];
  GsTables tb;
  gs_stage_tables(g, dyn, tb);
  Workspace ws;
  WalkScratch sc;
  wsp.carve(blockIdx.x, ws, sc);
  for (int job = blockIdx.x; job < 2 * B; job += gridDim.x) {
    int b = job >> 1;
    bool exact = job & 1;
    if (threadIdx.x == 0) {
      int m = 0;
      for (int j = 0; j < k; ++j) {
        int t = tok[(long long)b * k + j];
        if (t < 0) continue;
        s_pos[m] = pos[(long long)b * k + j];
        s_tok[m] = t;
        ++m;
      }
      ns = m;
    }
    __syncthreads();
    int r = -1;
    if (ns >= 2) {  // a set of at most one candidate is never tested
      Subst s{s_pos, s_tok, ns};
      if (exact) {
        EarleyColsGS<false> cols(g, tb, table, ws, sc, wsp.dims, sh, gss);
        cols.par = g.gs_par != 0;
        cols.wscr = (uint32_t*)(dyn + gs_tables_bytes(g.D, g.W, g.adv_steps));
        Walk<EarleyColsGS<false>> w(cols, g, table, sc, sh, vocab);
        r = w.run(x + (long long)b * n, n, s);
      } else {
        CoverCols cols(g, ws, wsp.dims, sh);
        Walk<CoverCols> w(cols, g, table, sc, sh, vocab);
        r = w.run(x + (long long)b * n, n, s);
      }
    }
    if (threadIdx.x == 0) spec[2 * b + (exact ? 1 : 0)] = (int8_t)(r == 1 ? 1 : (r == 0 ? 0 : -1));
    __syncthreads();
  }
}

__global__ void __launch_bounds__(kSelThreads) k_select(DevGrammar g, const LexEntry* __restrict__ table, int vocab,
                                                     const int32_t* __restrict__ x, int B, int n,
                                                     const int32_t* __restrict__ pos, int k,
                                                     const int32_t* __restrict__ tok, const float* __restrict__ conf,
                                                     uint8_t* __restrict__ selected, WsPack wsp,
                                                     const int8_t* __restrict__ spec, unsigned long long* stats) {
  __shared__ WalkShared sh;
  __shared__ GsShared gss;
  extern __shared__ __align__(16) unsigned char dyn[];
  GsTables tb;
  gs_stage_tables(g, dyn, tb);
  __shared__ int c_slot[kMaxSel], c_pos[kMaxSel], c_tok[kMaxSel];
  __shared__ int s_pos[kMaxSel], s_tok[kMaxSel];
  __shared__ SelFrame stack[2 * kMaxSel + 8];
  __shared__ int sp, nc, action, result, bad, overflow;
  __shared__ unsigned long long ret, final_set;
  Workspace ws;
  WalkScratch sc;
  wsp.carve(blockIdx.x, ws, sc);
  EarleyColsGS<false> ecols(g, tb, table, ws, sc, wsp.dims, sh, gss);
  ecols.par = g.gs_par != 0;
  ecols.wscr = (uint32_t*)(dyn + gs_tables_bytes(g.D, g.W, g.adv_steps));
  CoverCols ccols(g, ws, wsp.dims, sh);
  Walk<EarleyColsGS<false>> exact(ecols, g, table, sc, sh, vocab);
  Walk<CoverCols> cover(ccols, g, table, sc, sh, vocab);
  for (int b = blockIdx.x; b < B; b += gridDim.x) {
    const int32_t* xb = x + (long long)b * n;
    if (threadIdx.x == 0) {
      // C: proposed (position, token) pairs, by descending confidence then
      // ascending position (insertion sort; k <= 64)
      int m = 0;
      bad = 0;
      overflow = 0;
      for (int j = 0; j < k; ++j) {
        int t = tok[(long long)b * k + j];
        if (t < 0) continue;
        float cf = conf[(long long)b * k + j];
        if (cf != cf) bad = 1;
        int p = pos[(long long)b * k + j];
        int i = m++;
        while (i > 0) {
          float cp = conf[(long long)b * k + c_slot[i - 1]];
          if (cp > cf || (cp == cf && c_pos[i - 1] < p)) break;
          c_slot[i] = c_slot[i - 1];
          c_pos[i] = c_pos[i - 1];
          c_tok[i] = c_tok[i - 1];
          --i;
        }
        c_slot[i] = j;
        c_pos[i] = p;
        c_tok[i] = t;
      }
      nc = m;
      sp = 0;
      stack[0] = SelFrame{0, 0, 0ull, nc == 64 ? ~0ull : ((1ull << nc) - 1), 0ull, 0ull};
      sp = 1;
      final_set = 0;
      if (bad) sp = 0;
    }
    __syncthreads();
    for (;;) {
      // thread 0 advances the recursion until it needs a test or finishes
      if (threadIdx.x == 0) {
        action = 0;
        while (sp > 0 && action == 0) {
          if (sp >= 2 * kMaxSel + 6) {  // recursion deeper than Alg. 4 can go
            overflow = 1;
            sp = 0;
            break;
          }
          SelFrame& f = stack[sp - 1];
          unsigned long long set = f.set;
          // split in confidence order: first ceil(|set|/2) members
          auto halves = [&](unsigned long long s, unsigned long long& L, unsigned long long& R) {
            int cnt = __popcll(s), h = (cnt + 1) / 2;
            L = 0;
            unsigned long long r = s;
            for (int i = 0; i < h; ++i) {
              unsigned long long lo = r & (~r + 1);
              L |= lo;
              r &= r - 1;
            }
            R = s & ~L;
          };
          if (f.kind == 0) {
            if (f.pc == 0) {
              f.pc = 1;
              stack[sp++] = SelFrame{1, 0, 0ull, set, 0ull, 0ull};
            } else if (f.pc == 1) {
              f.pc = 2;
              stack[sp++] = SelFrame{2, 0, 0ull, ret, 0ull, 0ull};
            } else {
              final_set = ret;
              --sp;
            }
          } else if (f.kind == 1) {  // RelaxedSelect(x (+) base, set)
            if (f.pc == 0) {
              if (__popcll(set) <= 1) {
                ret = 0;
                --sp;
              } else {
                f.pc = 1;
                action = 1;  // cover test of base | set
                f.a = f.base | set;
              }
            } else if (f.pc == 1) {
              if (result == 1) {
                ret = set;
                --sp;
              } else {
                unsigned long long L, R;
                halves(set, L, R);
                f.a = R;
                f.pc = 2;
                stack[sp++] = SelFrame{1, 0, f.base, L, 0ull, 0ull};
              }
            } else if (f.pc == 2) {
              f.b = ret;
              f.pc = 3;
              unsigned long long R = f.a;
              stack[sp++] = SelFrame{1, 0, f.base | ret, R, 0ull, 0ull};
            } else {
              ret = f.b | ret;
              --sp;
            }
          } else {  // ExactShrink(x (+) base, set)
            if (f.pc == 0) {
              if (__popcll(set) <= 1) {
                ret = 0;
                --sp;
              } else {
                f.pc = 1;
                action = 2;  // exact joint check of base | set
                f.a = f.base | set;
              }
            } else if (f.pc == 1) {
              if (result == 1) {
                ret = set;
                --sp;
              } else {
                unsigned long long L, R;
                halves(set, L, R);
                f.a = R;
                f.pc = 2;
                stack[sp++] = SelFrame{2, 0, f.base, L, 0ull, 0ull};
              }
            } else if (f.pc == 2) {
              f.b = ret;  // B'_L
              f.pc = 3;
              stack[sp++] = SelFrame{1, 0, f.base | ret, f.a, 0ull, 0ull};
            } else if (f.pc == 3) {
              f.pc = 4;
              stack[sp++] = SelFrame{2, 0, f.base | f.b, ret, 0ull, 0ull};
            } else {
              ret = f.b | ret;
              --sp;
            }
          }
        }
        if (action != 0) {
          unsigned long long m = stack[sp - 1].a;
          int ns = 0;
          for (int i = 0; i < nc; ++i)
            if ((m >> i) & 1ull) {
              s_pos[ns] = c_pos[i];
              s_tok[ns] = c_tok[i];
              ++ns;
            }
          result = ns;  // substitution count for the test
        }
      }
      __syncthreads();
      int act = action;
      if (act == 0) break;
      Subst s{s_pos, s_tok, result};
      // the test of the whole candidate set was run ahead (k_select_spec)
      unsigned long long full = nc == 64 ? ~0ull : ((1ull << nc) - 1);
      int cached = (spec && stack[sp - 1].a == full) ? spec[2 * b + (act == 1 ? 0 : 1)] : -1;
      __syncthreads();
      int r = cached >= 0 ? cached : ((act == 1) ? cover.run(xb, n, s) : exact.run(xb, n, s));
      if (threadIdx.x == 0) {
        if (r < 0) {
          overflow |= (r == -1);
          bad |= (r == -2);
          sp = 0;
        }
        result = r == 1 ? 1 : 0;
        atomicAdd(&stats[act == 1 ? S_COVER : S_EXACT], 1ull);
      }
      __syncthreads();
    }
    if (threadIdx.x == 0) {
      for (int j = 0; j < k; ++j) selected[(long long)b * k + j] = overflow ? 2 : 0;
      if (!overflow && !bad) {
        for (int i = 0; i < nc; ++i)
          if ((final_set >> i) & 1ull) selected[(long long)b * k + c_slot[i]] = 1;
        atomicAdd(&stats[S_SELECTED], (unsigned long long)__popcll(final_set));
      }
      if (bad) atomicAdd(&stats[S_BAD], 1ull);
      if (overflow) atomicAdd(&stats[S_OVERFLOW], 1ull);
    }
    __syncthreads();
  }
}

// Alg. 1's sequential rejection fallback: fill = max(0, n_target[b] - |B|)
// more commits, each the highest-confidence candidate (ties: position, then
// candidate index) at a still-masked position that was not rejected and
// whose update passes the exact test (a whole-graph walk of x (+) c with the
// Gauss-Seidel columns); a candidate that fails is rejected for good (x only
// gains commits, and completability is monotone).  With the single-candidate
// bits of x before the commits (valid, may be null), a candidate whose bit
// is 0 is rejected without a walk: its test would fail.
//
// The loop runs in rounds, m CTAs per sequence: CTA s tests the s-th
// candidate of the current order against the current x, all at once; then
// the round is read in order, exactly as the sequential loop would meet
// it -- failed tests reject, the first passing one is committed, and after
// that commit a failed test still rejects (it fails against the larger x
// too) while a passing one is tested again next round.  The result is the
// sequential loop's; only the tests after a commit are spent.
//
// State per sequence (global): fb[0] commits still wanted, fb[1] active.

// per sequence: outputs cleared, rejections from the validity bits, the
// fill, bad inputs; counts the active sequences
__global__ void k_fallback_init(int B, int n, const int32_t* __restrict__ pos, int k,
                                const float* __restrict__ conf, int K, const int32_t* __restrict__ n_target,
                                const uint8_t* __restrict__ selected, const uint8_t* __restrict__ valid,
                                int32_t* __restrict__ filled, uint8_t* __restrict__ rej, int32_t* __restrict__ fb,
                                unsigned long long* __restrict__ active, unsigned long long* stats) {
  const int b = blockIdx.x;
  if (b >= B) return;
  const int nc = k * K;
  __shared__ int s_bad;
  if (threadIdx.x == 0) s_bad = 0;
  __syncthreads();
  for (int j = threadIdx.x; j < k; j += blockDim.x) {
    filled[(long long)b * k + j] = -1;
    const int p = pos[(long long)b * k + j];
    if (p < 0 || p >= n) s_bad = 1;
  }
  for (int q = threadIdx.x; q < nc; q += blockDim.x) {
    rej[(long long)b * nc + q] = (valid && valid[(long long)b * nc + q] == 0) ? 1 : 0;
    const float cf = conf[(long long)b * nc + q];
    if (cf != cf) s_bad = 1;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int nsel = 0;
    if (selected)
      for (int j = 0; j < k; ++j) nsel += selected[(long long)b * k + j] == 1;
    const int fill = n_target[b] - nsel;
    fb[2 * b] = fill;
    fb[2 * b + 1] = (!s_bad && fill > 0) ? 1 : 0;
    if (s_bad) atomicAdd(&stats[S_BAD], 1ull);
    if (fb[2 * b + 1]) atomicAdd(active, 1ull);
  }
}

// Block: the best candidate of sequence b (the order above) among those not
// rejected, at masked positions, and not in excl[0..nex); -1 if none.
__device__ int fallback_best(int b, const int32_t* xb, const int32_t* pos, int k, const float* conf, int K,
                             const uint8_t* rej, const int* excl, int nex, float* r_cf, int* r_q) {
  const int nc = k * K;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  auto before = [&](float ca, int qa, float cb, int qb) -> bool {  // (ca, qa) ahead of (cb, qb)
    if (qb < 0) return qa >= 0;
    if (qa < 0) return false;
    if (ca != cb) return ca > cb;
    const int pa = pos[(long long)b * k + qa / K], pb = pos[(long long)b * k + qb / K];
    return pa < pb || (pa == pb && qa < qb);
  };
  float bc = 0.f;
  int bq = -1;
  for (int q = threadIdx.x; q < nc; q += blockDim.x) {
    if (rej[(long long)b * nc + q]) continue;
    if (xb[pos[(long long)b * k + q / K]] >= 0) continue;  // committed by the selected batch or here
    bool ex = false;
    for (int i = 0; i < nex; ++i) ex |= excl[i] == q;
    if (ex) continue;
    const float cf = conf[(long long)b * nc + q];
    if (before(cf, q, bc, bq)) {
      bc = cf;
      bq = q;
    }
  }
  for (int off = 16; off; off >>= 1) {
    const float oc = __shfl_xor_sync(0xffffffffu, bc, off);
    const int oq = __shfl_xor_sync(0xffffffffu, bq, off);
    if (before(oc, oq, bc, bq)) {
      bc = oc;
      bq = oq;
    }
  }
  if (lane == 0) {
    r_cf[warp] = bc;
    r_q[warp] = bq;
  }
  __syncthreads();
  float c0 = 0.f;
  int q0 = -1;
  for (int i = 0; i < (int)(blockDim.x >> 5); ++i)
    if (before(r_cf[i], r_q[i], c0, q0)) {
      c0 = r_cf[i];
      q0 = r_q[i];
    }
  __syncthreads();
  return q0;
}

// One round: job (b, s) tests the s-th candidate of sequence b's order.
// res[(b m + s) 2] = candidate (-1: none), [+1] = 1 pass, 0 fail, -1 capacity.
__global__ void __launch_bounds__(kSelThreads) k_fallback_round(DevGrammar g, const LexEntry* __restrict__ table,
                                                             int vocab, const int32_t* __restrict__ x, int B, int n,
                                                             const int32_t* __restrict__ pos, int k,
                                                             const int32_t* __restrict__ cand,
                                                             const float* __restrict__ conf, int K, int m,
                                                             const uint8_t* __restrict__ rej,
                                                             const int32_t* __restrict__ fb, int32_t* __restrict__ res,
                                                             WsPack wsp, unsigned long long* stats) {
  __shared__ WalkShared sh;
  __shared__ GsShared gss;
  extern __shared__ __align__(16) unsigned char dyn[];
  GsTables tb;
  gs_stage_tables(g, dyn, tb);
  __shared__ float r_cf[kSelThreads / 32];
  __shared__ int r_q[kSelThreads / 32];
  __shared__ int excl[kMaxFallbackSpec];
  __shared__ int s_pos[1], s_tok[1];
  Workspace ws;
  WalkScratch sc;
  wsp.carve(blockIdx.x, ws, sc);
  EarleyColsGS<false> cols(g, tb, table, ws, sc, wsp.dims, sh, gss);
  cols.par = g.gs_par != 0;
  cols.wscr = (uint32_t*)(dyn + gs_tables_bytes(g.D, g.W, g.adv_steps));
  Walk<EarleyColsGS<false>> walk(cols, g, table, sc, sh, vocab);
  unsigned long long n_chk = 0;
  for (long long job = blockIdx.x; job < (long long)B * m; job += gridDim.x) {
    const int b = (int)(job / m), sl = (int)(job % m);
    int32_t* out = res + 2 * job;
    if (!fb[2 * b + 1]) {
      if (threadIdx.x == 0) {
        out[0] = -1;
        out[1] = 0;
      }
      continue;
    }
    const int32_t* xb = x + (long long)b * n;
    int q = -1;
    for (int i = 0; i <= sl; ++i) {
      q = fallback_best(b, xb, pos, k, conf, K, rej, excl, i, r_cf, r_q);
      if (q < 0) break;
      if (threadIdx.x == 0) excl[i] = q;
      __syncthreads();
    }
    if (q < 0) {
      if (threadIdx.x == 0) {
        out[0] = -1;
        out[1] = 0;
      }
      __syncthreads();
      continue;
    }
    if (threadIdx.x == 0) {
      s_pos[0] = pos[(long long)b * k + q / K];
      s_tok[0] = cand[(long long)b * k * K + q];
    }
    __syncthreads();
    Subst su{s_pos, s_tok, 1};
    const int r = walk.run(xb, n, su);
    if (threadIdx.x == 0) {
      out[0] = q;
      out[1] = r;
      ++n_chk;
    }
    __syncthreads();
  }
  if (threadIdx.x == 0 && n_chk) atomicAdd(&stats[S_FB_CHECKS], n_chk);
}

// One thread per sequence: read the round in order (see above); counts the
// sequences still active.
__global__ void k_fallback_resolve(int B, int32_t* __restrict__ x, int n, const int32_t* __restrict__ pos, int k,
                                   const int32_t* __restrict__ cand, int K, int m, uint8_t* __restrict__ rej,
                                   int32_t* __restrict__ fb, const int32_t* __restrict__ res,
                                   int32_t* __restrict__ filled, unsigned long long* __restrict__ active,
                                   unsigned long long* stats) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B || !fb[2 * b + 1]) return;
  const int nc = k * K;
  bool committed = false, any = false;
  unsigned long long n_com = 0, n_ovf = 0;
  for (int sl = 0; sl < m; ++sl) {
    const int q = res[2 * ((long long)b * m + sl)], r = res[2 * ((long long)b * m + sl) + 1];
    if (q < 0) break;
    any = true;
    if (!committed) {
      if (r == 1) {
        const int p = pos[(long long)b * k + q / K];
        const int t = cand[(long long)b * nc + q];
        x[(long long)b * n + p] = t;
        filled[(long long)b * k + q / K] = t;
        ++n_com;
        committed = true;
        if (--fb[2 * b] <= 0) fb[2 * b + 1] = 0;
      } else {
        rej[(long long)b * nc + q] = 1;
        if (r == -1) ++n_ovf;
      }
    } else if (r == 0) {
      rej[(long long)b * nc + q] = 1;  // fails against x, so against x with the commit
    }
  }
  if (!any) fb[2 * b + 1] = 0;  // every candidate rejected or its position committed
  if (n_com) atomicAdd(&stats[S_FB_COMMITS], n_com);
  if (n_ovf) atomicAdd(&stats[S_OVERFLOW], n_ovf);
  if (fb[2 * b + 1]) atomicAdd(active, 1ull);
}

namespace epic {

void launch_select_spec(dim3 grid, cudaStream_t st, const DevGrammar& g, const LexEntry* table, int vocab,
                        const int32_t* x, int B, int n, const int32_t* pos, int k, const int32_t* tok, int8_t* spec,
                        const WsPack& wsp) {
  const size_t dyn = gs_tables_bytes(g.D, g.W, g.adv_steps) + gs_warp_scratch_bytes();
  DevGrammar gg = g;
  gg.gs_par = gs_parallel_enabled(g.W);
  cudaFuncSetAttribute(k_select_spec, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
  k_select_spec<<<grid, kSelThreads, dyn, st>>>(gg, table, vocab, x, B, n, pos, k, tok, spec, wsp);
}

void launch_select(dim3 grid, cudaStream_t st, const DevGrammar& g, const LexEntry* table, int vocab,
                   const int32_t* x, int B, int n, const int32_t* pos, int k, const int32_t* tok, const float* conf,
                   uint8_t* selected, const WsPack& wsp, const int8_t* spec, unsigned long long* stats) {
  const size_t dyn = gs_tables_bytes(g.D, g.W, g.adv_steps) + gs_warp_scratch_bytes();
  DevGrammar gg = g;
  gg.gs_par = gs_parallel_enabled(g.W);
  cudaFuncSetAttribute(k_select, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
  k_select<<<grid, kSelThreads, dyn, st>>>(gg, table, vocab, x, B, n, pos, k, tok, conf, selected, wsp, spec, stats);
}

void launch_fallback_init(int B, cudaStream_t st, int n, const int32_t* pos, int k, const float* conf, int K,
                          const int32_t* n_target, const uint8_t* selected, const uint8_t* valid, int32_t* filled,
                          uint8_t* rej, int32_t* fb, unsigned long long* active, unsigned long long* stats) {
  k_fallback_init<<<B, 256, 0, st>>>(B, n, pos, k, conf, K, n_target, selected, valid, filled, rej, fb, active,
                                     stats);
}

void launch_fallback_round(dim3 grid, cudaStream_t st, const DevGrammar& g, const LexEntry* table, int vocab,
                           const int32_t* x, int B, int n, const int32_t* pos, int k, const int32_t* cand,
                           const float* conf, int K, int m, const uint8_t* rej, const int32_t* fb, int32_t* res,
                           const WsPack& wsp, unsigned long long* stats) {
  const size_t dyn = gs_tables_bytes(g.D, g.W, g.adv_steps) + gs_warp_scratch_bytes();
  DevGrammar gg = g;
  gg.gs_par = gs_parallel_enabled(g.W);
  cudaFuncSetAttribute(k_fallback_round, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
  k_fallback_round<<<grid, kSelThreads, dyn, st>>>(gg, table, vocab, x, B, n, pos, k, cand, conf, K, m, rej, fb, res,
                                                wsp, stats);
}

void launch_fallback_resolve(int B, cudaStream_t st, int32_t* x, int n, const int32_t* pos, int k,
                             const int32_t* cand, int K, int m, uint8_t* rej, int32_t* fb, const int32_t* res,
                             int32_t* filled, unsigned long long* active, unsigned long long* stats) {
  k_fallback_resolve<<<(B + 127) / 128, 128, 0, st>>>(B, x, n, pos, k, cand, K, m, rej, fb, res, filled, active,
                                                      stats);
}

}  // namespace epic
