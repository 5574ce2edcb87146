// Alg. 4 (relaxed compatible-subset selection with exact re-check): kernels
// and launchers.
#include <cuda_runtime.h>

#include "launch.h"

using namespace epic;

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
__global__ void __launch_bounds__(kThreads) k_select_spec(DevGrammar g, const LexEntry* __restrict__ table, int vocab,
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

__global__ void __launch_bounds__(kThreads) k_select(DevGrammar g, const LexEntry* __restrict__ table, int vocab,
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

// Alg. 1's sequential rejection fallback, one CTA per sequence: fill =
// max(0, n_target[b] - |B|) more commits, each the highest-confidence
// candidate (ties: position, then candidate index) at a still-masked
// position that was not rejected and whose update passes the exact test
// (a whole-graph walk of x (+) c with the Gauss-Seidel columns); a candidate
// that fails is rejected for good (x only gains commits, and completability
// is monotone).  With the single-candidate bits of x before the commits
// (valid, may be null), a candidate whose bit is 0 is rejected without a
// walk: its test would fail (monotonicity again).  Commits go straight into
// x.  Bounded by the k K candidates.
__global__ void __launch_bounds__(kThreads) k_fallback(DevGrammar g, const LexEntry* __restrict__ table, int vocab,
                                                       int32_t* __restrict__ x, int B, int n,
                                                       const int32_t* __restrict__ pos, int k,
                                                       const int32_t* __restrict__ cand,
                                                       const float* __restrict__ conf, int K,
                                                       const int32_t* __restrict__ n_target,
                                                       const uint8_t* __restrict__ selected,
                                                       const uint8_t* __restrict__ valid,
                                                       int32_t* __restrict__ filled, WsPack wsp,
                                                       unsigned long long* stats) {
  __shared__ WalkShared sh;
  __shared__ GsShared gss;
  extern __shared__ __align__(16) unsigned char dyn[];
  GsTables tb;
  gs_stage_tables(g, dyn, tb);
  __shared__ uint8_t rej[kMaxFallbackCand];
  __shared__ float r_cf[kThreads / 32];
  __shared__ int r_q[kThreads / 32];
  __shared__ int s_pos[1], s_tok[1];
  __shared__ int s_fill, s_bad, s_q;
  Workspace ws;
  WalkScratch sc;
  wsp.carve(blockIdx.x, ws, sc);
  EarleyColsGS<false> cols(g, tb, table, ws, sc, wsp.dims, sh, gss);
  Walk<EarleyColsGS<false>> walk(cols, g, table, sc, sh, vocab);
  const int nc = k * K;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  unsigned long long n_chk = 0, n_com = 0, n_ovf = 0, n_bad = 0;
  for (int b = blockIdx.x; b < B; b += gridDim.x) {
    int32_t* xb = x + (long long)b * n;
    for (int j = threadIdx.x; j < k; j += blockDim.x) filled[(long long)b * k + j] = -1;
    for (int q = threadIdx.x; q < nc; q += blockDim.x) rej[q] = (valid && valid[(long long)b * nc + q] == 0) ? 1 : 0;
    if (threadIdx.x == 0) {
      int nsel = 0;
      if (selected)
        for (int j = 0; j < k; ++j) nsel += selected[(long long)b * k + j] == 1;
      s_fill = n_target[b] - nsel;
      s_bad = 0;
      for (int q = 0; q < nc; ++q) {
        const float cf = conf[(long long)b * nc + q];
        if (cf != cf) s_bad = 1;
        const int p = pos[(long long)b * k + q / K];
        if (p < 0 || p >= n) s_bad = 1;
      }
    }
    __syncthreads();
    if (s_bad) {
      if (threadIdx.x == 0) ++n_bad;
      continue;
    }
    int done = 0;
    for (int guard = 0; guard <= nc && done < s_fill; ++guard) {
      // the next candidate: highest confidence, then lowest position, then
      // lowest candidate index, among those not rejected at masked positions
      float bc = 0.f;
      int bq = -1;
      for (int q = threadIdx.x; q < nc; q += blockDim.x) {
        if (rej[q]) continue;
        const int p = pos[(long long)b * k + q / K];
        if (xb[p] >= 0) continue;  // committed by the selected batch or earlier here
        const float cf = conf[(long long)b * nc + q];
        const bool better = bq < 0 || cf > bc ||
                            (cf == bc && (p < pos[(long long)b * k + bq / K] ||
                                          (p == pos[(long long)b * k + bq / K] && q < bq)));
        if (better) {
          bc = cf;
          bq = q;
        }
      }
      for (int off = 16; off; off >>= 1) {
        const float oc = __shfl_xor_sync(0xffffffffu, bc, off);
        const int oq = __shfl_xor_sync(0xffffffffu, bq, off);
        bool take = false;
        if (oq >= 0) {
          if (bq < 0 || oc > bc) {
            take = true;
          } else if (oc == bc) {
            const int po = pos[(long long)b * k + oq / K], pb = pos[(long long)b * k + bq / K];
            take = po < pb || (po == pb && oq < bq);
          }
        }
        if (take) {
          bc = oc;
          bq = oq;
        }
      }
      if (lane == 0) {
        r_cf[warp] = bc;
        r_q[warp] = bq;
      }
      __syncthreads();
      if (threadIdx.x == 0) {
        float c0 = 0.f;
        int q0 = -1;
        for (int i = 0; i < (int)(blockDim.x >> 5); ++i) {
          const int oq = r_q[i];
          if (oq < 0) continue;
          const float oc = r_cf[i];
          bool take = q0 < 0 || oc > c0;
          if (!take && oc == c0) {
            const int po = pos[(long long)b * k + oq / K], pb = pos[(long long)b * k + q0 / K];
            take = po < pb || (po == pb && oq < q0);
          }
          if (take) {
            c0 = oc;
            q0 = oq;
          }
        }
        s_q = q0;
        if (q0 >= 0) {
          s_pos[0] = pos[(long long)b * k + q0 / K];
          s_tok[0] = cand[(long long)b * nc + q0];
        }
      }
      __syncthreads();
      const int q = s_q;
      if (q < 0) break;  // every candidate rejected
      Subst su{s_pos, s_tok, 1};
      const int r = walk.run(xb, n, su);
      if (threadIdx.x == 0) {
        ++n_chk;
        if (r == 1) {
          xb[s_pos[0]] = s_tok[0];
          filled[(long long)b * k + q / K] = s_tok[0];
          ++n_com;
        } else {
          rej[q] = 1;
          if (r == -1) ++n_ovf;
        }
      }
      __syncthreads();
      if (r == 1) ++done;
    }
  }
  if (threadIdx.x == 0) {
    atomicAdd(&stats[S_FB_CHECKS], n_chk);
    atomicAdd(&stats[S_FB_COMMITS], n_com);
    atomicAdd(&stats[S_OVERFLOW], n_ovf);
    atomicAdd(&stats[S_BAD], n_bad);
  }
}

namespace epic {

void launch_select_spec(dim3 grid, cudaStream_t st, const DevGrammar& g, const LexEntry* table, int vocab,
                        const int32_t* x, int B, int n, const int32_t* pos, int k, const int32_t* tok, int8_t* spec,
                        const WsPack& wsp) {
  const size_t dyn = gs_tables_bytes(g.D, g.W, g.adv_steps);
  cudaFuncSetAttribute(k_select_spec, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
  k_select_spec<<<grid, kThreads, dyn, st>>>(g, table, vocab, x, B, n, pos, k, tok, spec, wsp);
}

void launch_select(dim3 grid, cudaStream_t st, const DevGrammar& g, const LexEntry* table, int vocab,
                   const int32_t* x, int B, int n, const int32_t* pos, int k, const int32_t* tok, const float* conf,
                   uint8_t* selected, const WsPack& wsp, const int8_t* spec, unsigned long long* stats) {
  const size_t dyn = gs_tables_bytes(g.D, g.W, g.adv_steps);
  cudaFuncSetAttribute(k_select, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
  k_select<<<grid, kThreads, dyn, st>>>(g, table, vocab, x, B, n, pos, k, tok, conf, selected, wsp, spec, stats);
}

void launch_fallback(dim3 grid, cudaStream_t st, const DevGrammar& g, const LexEntry* table, int vocab, int32_t* x,
                     int B, int n, const int32_t* pos, int k, const int32_t* cand, const float* conf, int K,
                     const int32_t* n_target, const uint8_t* selected, const uint8_t* valid, int32_t* filled,
                     const WsPack& wsp, unsigned long long* stats) {
  const size_t dyn = gs_tables_bytes(g.D, g.W, g.adv_steps);
  cudaFuncSetAttribute(k_fallback, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
  k_fallback<<<grid, kThreads, dyn, st>>>(g, table, vocab, x, B, n, pos, k, cand, conf, K, n_target, selected, valid,
                                          filled, wsp, stats);
}

}  // namespace epic
