// The per-sequence arena of checks by region: the forward chart of x, its
// recorded graph, and the tables of the good pass.
#pragma once
#include "walk.cuh"
#include "warpwalk.cuh"

namespace epic {

// Per-sequence forward chart and its tables.
struct SeqArena {
  WWs ws;          // the forward walk's workspace; org/bits/esum/col_off are the chart
  SeqRec rec;
  uint32_t* good;      // [emax][W]
  int32_t* last_col;   // [nmax] last column holding origin u (-1: none)
  int32_t* in_off;     // [nmax + 1] edges are stored by target column
  int32_t* out_off;    // [nmax + 1]
  int32_t* out_idx;    // [edge_cap]
  int32_t* succ_off;   // [nmax + 1] columns holding origin u, ascending
  int32_t* succ_idx;   // [emax]
  uint32_t* expn;      // [nmax][W] scratch of the good pass
  int32_t* eidx;       // [nmax (nmax + 1) / 2] entry of (column j, origin o <= j), -1: none
  uint8_t* gnz;        // [emax] the entry has a good item
  int32_t* cursor;     // [2 (nmax + 1)] scratch of the good pass
  int32_t* key_q;      // [kMaxQ] scratch of the block forward walk
  uint32_t* bexpn;     // [nmax][W]
  uint32_t* bnew;      // [nmax][VW]
};

struct SeqPack {
  char* base;
  size_t per_seq;
  int nmax, n, W, VW, edge_cap;
  long long emax;
  __host__ __device__ static size_t r(size_t b) { return (b + 255) & ~(size_t)255; }
  __host__ __device__ size_t bytes() const {
    size_t nm = nmax;
    return r(nm * W * 4) + r(nm * VW * 4) + r((nm + 1) * 4) + 7 * r(kWMaxQ * 4) + r(kWMaxQ * 16) + r(kWMaxQ * 32) +
           r(nm * 8) + r((size_t)emax * 4) + r((size_t)emax * 8) + r((size_t)emax * W * 4)  // WWs
           + r(nm) + 2 * r((size_t)edge_cap * 4) + r((size_t)edge_cap * 32) + 3 * r((size_t)n * 4) +
           r((size_t)emax * VW * 4) + r(32)                                                 // SeqRec
           + r((size_t)emax * W * 4) + r(nm * 4) + 3 * r((nm + 1) * 4) + r((size_t)edge_cap * 4) +
           r((size_t)emax * 4) + r(nm * W * 4) + r(nm * (nm + 1) / 2 * 4) + r((size_t)emax) + r(2 * (nm + 1) * 4) + r(kMaxQ * 4) +
           r(nm * W * 4) + r(nm * VW * 4);
  }
  __device__ SeqArena carve(long long b) const {
    SeqArena a;
    char* p = base + per_seq * (size_t)b;
    auto take = [&](size_t bytes) {
      char* q = p;
      p += r(bytes);
      return q;
    };
    size_t nm = nmax;
    a.ws.stage = (uint32_t*)take(nm * W * 4);
    a.ws.bdone = (uint32_t*)take(nm * VW * 4);
    a.ws.col_off = (int32_t*)take((nm + 1) * 4);
    a.ws.f_q = (int32_t*)take(kWMaxQ * 4);
    a.ws.f_c = (int32_t*)take(kWMaxQ * 4);
    a.ws.g_src = (int32_t*)take(kWMaxQ * 4);
    a.ws.g_end = (int32_t*)take(kWMaxQ * 4);
    a.ws.g_len = (int32_t*)take(kWMaxQ * 4);
    a.ws.g_last = (int32_t*)take(kWMaxQ * 4);
    a.ws.key_q = (int32_t*)take(kWMaxQ * 4);
    a.ws.g_tail = (uint32_t*)take(kWMaxQ * 16);
    a.ws.g_lbl = (uint32_t*)take(kWMaxQ * 32);
    a.ws.ssum = (uint32_t*)take(nm * 8);
    a.ws.org = (int32_t*)take((size_t)emax * 4);
    a.ws.esum = (uint32_t*)take((size_t)emax * 8);
    a.ws.bits = (uint32_t*)take((size_t)emax * W * 4);
    a.rec.col_gap = (uint8_t*)take(nm);
    a.rec.e_dst = (int32_t*)take((size_t)edge_cap * 4);
    a.rec.e_src = (int32_t*)take((size_t)edge_cap * 4);
    a.rec.e_lbl = (uint32_t*)take((size_t)edge_cap * 32);
    a.rec.gap_col = (int32_t*)take((size_t)n * 4);
    a.rec.pre_col = (int32_t*)take((size_t)n * 4);
    a.rec.post_col = (int32_t*)take((size_t)n * 4);
    a.rec.cnt = (uint32_t*)take((size_t)emax * VW * 4);
    a.rec.meta = (int32_t*)take(32);
    a.rec.edge_cap = edge_cap;
    a.rec.n_edges = 0;
    a.good = (uint32_t*)take((size_t)emax * W * 4);
    a.last_col = (int32_t*)take(nm * 4);
    a.in_off = (int32_t*)take((nm + 1) * 4);
    a.out_off = (int32_t*)take((nm + 1) * 4);
    a.succ_off = (int32_t*)take((nm + 1) * 4);
    a.out_idx = (int32_t*)take((size_t)edge_cap * 4);
    a.succ_idx = (int32_t*)take((size_t)emax * 4);
    a.expn = (uint32_t*)take(nm * W * 4);
    a.eidx = (int32_t*)take(nm * (nm + 1) / 2 * 4);
    a.gnz = (uint8_t*)take((size_t)emax);
    a.cursor = (int32_t*)take(2 * (nm + 1) * 4);
    a.key_q = (int32_t*)take(kMaxQ * 4);
    a.bexpn = (uint32_t*)take(nm * W * 4);
    a.bnew = (uint32_t*)take(nm * VW * 4);
    return a;
  }
};

// meta slots of a sequence's record
enum { M_NCOLS = 0, M_NEDGES = 1, M_START = 2, M_ACCEPT = 3, M_STATUS = 4, M_NENT = 5 };

}  // namespace epic
