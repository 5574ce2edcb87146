// Checks by region, step 3: one warp per check walks only the candidate's
// region over the sequence's forward chart (see region.cuh).
#pragma once
#include "region.cuh"

namespace epic {

// ------------------------------------------------------------------ 3. checks by region
template <bool SM>
struct RegionCheck {
  WarpWalker<SM, true>& w;
  SeqArena& a;
  int32_t* fmap;     // [nmax] F node -> own column with carried rows (-1)
  int32_t* act;      // [nmax] own columns whose rows wait on nonterminals
  int32_t* act_f;    // [nmax] their F node

  // x (+) {(i, t)}: 1 valid, 0 invalid, -1 capacity
  __device__ int run(const int32_t* x, int n, int i, int t) {
    const int lane = threadIdx.x & 31;
    const int32_t* meta = a.rec.meta;
    const int NF = meta[M_NCOLS];
    // base chart
    w.base_cols = NF;
    w.base_ent = a.ws.col_off[NF];
    w.b_col_off = a.ws.col_off;
    w.b_org = a.ws.org;
    w.b_bits = a.ws.bits;
    w.b_esum = a.ws.esum;
    w.good = a.good;
    w.b_eidx = a.eidx;
    w.accept_node = meta[M_ACCEPT];
    w.ncols = NF;
    w.nent = 0;
    w.status = 0;
    w.nf = 0;
    w.found = 0;
    w.suffix_mode = false;
    w.region_start = -1;
    if (lane == 0) w.ws.col_off[0] = 0;
    __syncwarp();
    // the mask run [ra, rb] holding i
    int ra = i, rb = i;
    while (ra > 0 && x[ra - 1] < 0) --ra;
    while (rb + 1 < n && x[rb + 1] < 0) ++rb;
    int start = meta[M_START];
    int src;
    bool at_begin;
    int left_lo = 0, left_hi = 0;  // fixed tokens before t in the span
    if (i > ra) {
      src = a.rec.gap_col[i];  // the left part of the run is the whole run's gap
      at_begin = false;
    } else if (ra > 0) {
      int s = ra - 1;
      while (s > 0 && x[s - 1] >= 0) --s;
      src = a.rec.pre_col[ra - 1];
      at_begin = s == 0;
      left_lo = s;
      left_hi = ra;
    } else {  // t starts the output: a BEGIN node of the check's own
      int c = w.open_column();
      if (c < 0) return -1;
      w.seed(c);
      w.close_column(c, false);
      w.finish_column(c);
      if (w.status) return -1;
      src = c;
      at_begin = true;
      start = c;
      w.region_start = c;
    }
    int right_lo = 0, right_hi = 0;
    bool to_end;
    int rf;  // F node after the region
    if (i < rb) {
      to_end = false;
      rf = a.rec.gap_col[i];
    } else if (rb + 1 < n) {
      int e = rb + 1;
      while (e + 1 < n && x[e + 1] >= 0) ++e;
      right_lo = rb + 1;
      right_hi = e + 1;
      to_end = (e == n - 1);
      rf = to_end ? -1 : a.rec.post_col[rb + 1];
    } else {
      to_end = true;
      rf = -1;
    }
    w.start_col = start;
    w.frontier_from(src, at_begin);
    for (int p = left_lo; p < left_hi && w.nf > 0; ++p)
      if (!w.span_step(x[p])) return -1;
    // the region's last span step feeds the gap after it (unless the region
    // runs to the end): its end nodes reached by epsilon need no closure
    w.defer_to_gap = !to_end && right_hi == right_lo;
    const bool ok_t = w.nf == 0 || w.span_step(t);
    w.defer_to_gap = false;
    if (!ok_t) return -1;
    for (int p = right_lo; p < right_hi && w.nf > 0; ++p) {
      w.defer_to_gap = !to_end && p + 1 == right_hi;
      const bool ok = w.span_step(x[p]);
      w.defer_to_gap = false;
      if (!ok) return -1;
    }
    if (w.nf == 0) return 0;
    if (to_end) {
      int c = w.end_from_frontier();
      if (c < 0) return -1;
      w.close_column(c, false);
      w.finish_column(c);
      if (w.status) return -1;
      return w.accepts(c, start) ? 1 : 0;
    }
    // the node after the region, then the suffix, carrying only the items
    // whose origin is a node of the region
    for (int j = lane; j < NF; j += 32) fmap[j] = -1;
    __syncwarp();
    int nact = 0;
    w.suffix_mode = true;
    w.res_node = rf;
    {
      int c = w.gap_from_frontier();
      if (c < 0) return -1;
      w.close_column(c, true);
      w.finish_column(c);
      if (w.status) return -1;
      if (w.found) return 1;
      if (!w.column_empty(c)) {
        if (lane == 0) {
          fmap[rf] = c;
          act[0] = c;
          act_f[0] = rf;
        }
        __syncwarp();
        nact = 1;
      }
    }
    if (nact == 0) return 0;  // nothing of the region passes the node after it (a gap)
#ifdef EPIC_PHASE_TIMERS
    long long t_suffix = clock64();
#endif
    for (int j = rf + 1; j < NF; ++j) {
#ifdef EPIC_PHASE_TIMERS
      if (lane == 0) atomicAdd(&g_phase[12], 1ull);  // suffix columns walked
#endif
      int c = w.open_column();
      if (c < 0) return -1;
      w.res_node = j;
      // arrivals along F's edges into j from nodes that carry rows
      for (int e = a.in_off[j]; e < a.in_off[j + 1]; ++e) {
        int oc = fmap[a.rec.e_src[e]];
        if (oc < 0) continue;
        const uint32_t* L = a.rec.e_lbl + (size_t)e * 8;
        bool eps = true;
        for (int lw = 0; lw < 8; ++lw) eps &= L[lw] == 0;
        if (eps) {
          w.arrive(oc, nullptr, false);
        } else {
          w.label_set(L);
          w.arrive(oc, w.sh.lbl, true);
        }
      }
      // nested constituents from an earlier carrying node u completing at j
      for (int ai = 0; ai < nact; ++ai) {
        int u = act[ai], uf = act_f[ai];
        long long kc = w.find_base(j, uf);
        if (kc < 0) continue;
        for (int v = lane; v < w.VW; v += 32) w.sh.nt[v] = a.rec.cnt[(size_t)kc * w.VW + v];
        __syncwarp();
        uint32_t fold = 0;
        for (int v = 0; v < w.VW; ++v) fold |= w.sh.nt[v];
        if (!fold) continue;
        expn_of_set(w.g, w.sh.nt, w.sh.expn);
        __syncwarp();
        w.col_labelled = true;  // new items to close, not a copy of a closed column
        w.scatter(u, w.sh.expn, true, 0, fold);
        if (w.status) return -1;
      }
      w.close_column(c, a.rec.col_gap[j] != 0);
      w.finish_column(c);
      if (w.status) return -1;
      if (w.found) return 1;
      bool keep = !w.column_empty(c);
      if (keep && lane == 0) fmap[j] = c;
      // carrying nodes whose F origin can no longer complete anything retire
      int na = 0;
      for (int ai = 0; ai < nact; ++ai) {
        int uf = act_f[ai];
        if (a.last_col[uf] > j) {
          if (lane == 0) {
            act[na] = act[ai];
            act_f[na] = uf;
          }
          ++na;
        }
      }
      if (keep && a.last_col[j] > j) {
        if (lane == 0) {
          act[na] = c;
          act_f[na] = j;
        }
        ++na;
      }
      __syncwarp();
      nact = na;
      // a gap is a cut of the graph: if nothing is carried through it and no
      // earlier node can still complete past it, nothing of the region comes back
      if (!keep && a.rec.col_gap[j] && nact == 0) break;
    }
#ifdef EPIC_PHASE_TIMERS
    if (lane == 0) {
      atomicAdd(&g_phase[13], (unsigned long long)(clock64() - t_suffix));
      atomicAdd(&g_phase[14], 1ull);  // checks that reached the suffix walk
    }
#endif
    return w.found ? 1 : 0;
  }
};

// per-warp tables of a region check
struct RegScratch {
  int32_t* fmap;
  int32_t* act;
  int32_t* act_f;
};

template <bool SM>
__global__ void __launch_bounds__(32 * kWarpsPerCta) k_check(
    DevGrammar g, const LexEntry* __restrict__ table, int vocab, const int32_t* __restrict__ x, int n,
    const int32_t* __restrict__ pos, int k, const int32_t* __restrict__ cand, int K, long long total,
    uint8_t* __restrict__ valid, SeqPack sp, WPack wp, int32_t* __restrict__ regs, int rmax,
    unsigned long long* counter, unsigned long long* stats) {
  __shared__ WSh shm[kWarpsPerCta];
  extern __shared__ __align__(16) unsigned char dyn[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  WSh& sh = shm[warp];
  for (int w = lane; w < kWCols / 32; w += 32) {
    sh.touched[w] = 0;
    sh.dirty[w] = 0;
  }
  for (int v = lane; v < kWMaxVW; v += 32) {
    sh.vset[v] = 0;
    sh.vdone[v] = 0;
  }
  __syncwarp();
  const long long gw = (long long)blockIdx.x * (blockDim.x >> 5) + warp;
  WarpWalker<SM, true> walk(g, table, wp.carve(gw), sh, wp.nmax, wp.emax, vocab);
  if constexpr (SM) {
    size_t per = smem_per_warp(wp.nmax, rmax, g.W, g.VW);
    unsigned char* base = dyn + per * warp;
    uint32_t* rows = (uint32_t*)base;
    uint32_t* bd = rows + (size_t)rmax * g.W;
    int32_t* sorg = (int32_t*)(bd + (size_t)rmax * g.VW);
    uint32_t* ssum = (uint32_t*)(sorg + rmax);
    int16_t* so = (int16_t*)(ssum + 2 * rmax);
    walk.set_smem(rows, bd, so, sorg, ssum, rmax);
  }
  RegScratch rs;
  rs.fmap = regs + (size_t)gw * 3 * wp.nmax;
  rs.act = rs.fmap + wp.nmax;
  rs.act_f = rs.act + wp.nmax;
  unsigned long long n_checks = 0, n_valid = 0, n_ovf = 0, n_bad = 0, n_cols = 0, n_ent = 0;
  for (;;) {
    long long jb = 0;
    if (lane == 0) jb = (long long)atomicAdd(counter, 1ull);
    jb = __shfl_sync(0xffffffffu, jb, 0);
    if (jb >= total) break;
    long long b = jb / ((long long)k * K);
    long long jj = (jb / K) % k;
    const int32_t* xb = x + b * n;
    int i = pos[b * k + jj], t = cand[jb];
    int r;
    long long own_cols = 0, own_ent = 0;  // columns and entries this check stored
    if (i < 0 || i >= n || xb[i] >= 0 || t < 0 || t >= vocab) {
      r = -2;
    } else {
      SeqArena a = sp.carve(b);
      int fs = a.rec.meta[M_STATUS];
      if (fs == 0) {
        r = 0;  // x is not completable, so no update of it is
      } else if (fs == 1) {
        RegionCheck<SM> rc{walk, a, rs.fmap, rs.act, rs.act_f};
        r = rc.run(xb, n, i, t);
        if (r < 0) walk.cleanup();
        own_cols = walk.ncols - walk.base_cols;
        own_ent = walk.nent;
      } else {  // the sequence's forward chart did not fit: walk the whole check
        walk.base_cols = 0;
        walk.base_ent = 0;
        walk.suffix_mode = false;
        r = walk.run(xb, n, i, t);
        own_cols = walk.ncols;
        own_ent = walk.nent;
      }
      walk.base_cols = 0;
      walk.base_ent = 0;
      walk.suffix_mode = false;
    }
    if (lane == 0) valid[jb] = r == 1 ? 1 : (r == -1 ? 2 : 0);
    ++n_checks;
    n_valid += r == 1;
    n_ovf += r == -1;
    n_bad += r == -2;
    n_cols += own_cols;
    n_ent += own_ent;
  }
  if (lane == 0 && n_checks) {
    atomicAdd(&stats[0], n_checks);
    atomicAdd(&stats[1], n_valid);
    atomicAdd(&stats[2], n_ovf);
    atomicAdd(&stats[3], n_bad);
    atomicAdd(&stats[4], n_cols);
    atomicAdd(&stats[5], n_ent);
  }
}

}  // namespace epic
