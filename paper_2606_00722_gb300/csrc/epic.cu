// Kernels and C-ABI of the EPIC hot path on sm_103a (see include/epic.h).
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <functional>
#include <mutex>
#include <new>
#include <stdexcept>
#include <string>
#include <vector>

#include "../../include/epic.h"
#include "../../include/epic_measure.h"
#include "grammar.h"
#include "launch.h"

using namespace epic;

// ================================================================ kernels

// K1: memoized lex table.  One thread per (token, entry state); consecutive
// threads share a token (its bytes are a broadcast read) and write
// consecutive 16-byte entries.
__global__ void k_lex_table(const int32_t* __restrict__ tok_off, const uint8_t* __restrict__ bytes, int vocab,
                            int Q, const int32_t* __restrict__ dfa_next, const int16_t* __restrict__ dfa_acc,
                            const uint8_t* __restrict__ skip, LexEntry* __restrict__ table, int* overflow) {
  long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (long long)vocab * Q) return;
  int t = (int)(idx / Q), q = (int)(idx % Q);
  bool ovf = false;
  const LexEntry e = lex_transduce(bytes, tok_off[t], tok_off[t + 1], q, dfa_next, dfa_acc, skip, &ovf);
  if (ovf) atomicExch(overflow, 1);
  table[idx] = e;
}

// Per proposed position: the highest-confidence candidate with valid bit 1.
__global__ void k_pick(const int32_t* __restrict__ cand, const float* __restrict__ conf,
                       const uint8_t* __restrict__ valid, int B, int k, int K, int32_t* __restrict__ tok,
                       float* __restrict__ out_conf) {
  long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (long long)B * k) return;
  int best = -1;
  float bc = 0.f;
  for (int c = 0; c < K; ++c) {
    long long q = i * K + c;
    if (valid[q] != 1) continue;
    float v = conf[q];
    if (best < 0 || v > bc) {
      best = c;
      bc = v;
    }
  }
  tok[i] = best < 0 ? -1 : cand[i * K + best];
  out_conf[i] = best < 0 ? 0.f : bc;
}

__global__ void k_commit(int32_t* __restrict__ x, int B, int n, const int32_t* __restrict__ pos, int k,
                         const int32_t* __restrict__ tok, const uint8_t* __restrict__ sel) {
  long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (long long)B * k) return;
  if (sel[i] != 1) return;
  long long b = i / k;
  int p = pos[i];
  if (p >= 0 && p < n) x[b * n + p] = tok[i];
}

// ================================================================ host side

struct epic_grammar {
  int device = 0;
  GrammarTables tabs;
  LexerDFA dfa;
  CoverTables cov;
  DevGrammar dg{};
  std::vector<void*> dev_allocs;
};

struct epic_lexer_table {
  const epic_grammar* g = nullptr;
  int vocab = 0;
  LexEntry* d_table = nullptr;  // dense tables; null for lazy ones
  // the grammar's device tables with this table's lazy memo (keys null: dense)
  DevGrammar dgl{};
  uint32_t* d_lz_keys = nullptr;  // lazy memo (Alg. 2's cache filled on use)
  uint32_t* d_lz_ready = nullptr;
  LexEntry* d_lz_vals = nullptr;
  int32_t* d_lz_off = nullptr;
  uint8_t* d_lz_bytes = nullptr;
  long long lz_cap = 0;
  char* d_ws = nullptr;
  size_t ws_bytes = 0;
  WsDims dims{};
  int ctas = 0;
  unsigned long long* d_stats = nullptr;
  mutable unsigned long long n_region = 0, n_vkernels = 0;  // host-side counters
  unsigned long long* d_counter = nullptr;
  int8_t* d_spec = nullptr;  // speculative Alg. 4 answers, 2 per sequence
  char* d_seq = nullptr;     // per-sequence forward charts (region checks)
  size_t seq_bytes = 0;
  int32_t* d_regs = nullptr; // per-warp tables of region checks
  char* d_wit = nullptr;     // witness extraction: goals and stack per sequence
  size_t wit_bytes = 0;
  char* d_fb = nullptr;      // rejection fallback: rejections, state and round results per sequence
  size_t fb_bytes = 0;
  mutable unsigned long long n_fb_rounds = 0;  // host-side counter: fallback rounds launched
  size_t regs_bytes = 0;
  int spec_cap = 0;
  char* d_wws = nullptr;   // warp-walk workspace
  size_t wws_bytes = 0;
  int wnmax = 0;
  long long wemax = 0;
  int wwarps = 0;
  cudaStream_t last = nullptr;
  // CUDA events around the kernels of the last epic_validate_batch call
  // (epic_last_kernel_times): kev[i] .. kev[i + 1] is kernel i
  cudaEvent_t kev[4] = {nullptr, nullptr, nullptr, nullptr};
  int nk = 0;
  const char* kname[3] = {nullptr, nullptr, nullptr};
  // the same around the two kernels of the last epic_select_compatible_subset
  cudaEvent_t sev[3] = {nullptr, nullptr, nullptr};
  bool sel_timed = false;
};

namespace {
// record event i of the table's kernel timing on st (created on first use)
void mark_event(cudaEvent_t* e, cudaStream_t st) {
  if (!*e && cudaEventCreate(e) != cudaSuccess) *e = nullptr;
  if (*e) cudaEventRecord(*e, st);
}
void mark(epic_lexer_table* t, int i, cudaStream_t st) { mark_event(&t->kev[i], st); }
}  // namespace

namespace {

template <class T>
epic_status upload(epic_grammar* g, const std::vector<T>& v, const T** out) {
  void* p = nullptr;
  size_t bytes = std::max<size_t>(sizeof(T), v.size() * sizeof(T));
  if (cudaMalloc(&p, bytes) != cudaSuccess) return EPIC_ERR_OOM;
  g->dev_allocs.push_back(p);
  if (!v.empty() && cudaMemcpy(p, v.data(), v.size() * sizeof(T), cudaMemcpyHostToDevice) != cudaSuccess)
    return EPIC_ERR_CUDA;
  *out = (const T*)p;
  return EPIC_OK;
}

int sm_count() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : 1;
}

// Default budget of one device workspace: a share of the GPU's memory, and no
// more than is free now plus what the workspace already holds (it is freed
// before it grows), less 1 GiB of headroom.  An environment variable (MiB)
// overrides.  The three workspaces (per-sequence charts 30 %, warp walks
// 25 %, block walks 25 %) leave a fifth of the GPU to the caller.
size_t workspace_budget(const char* env, double share, size_t held) {
  if (const char* e = getenv(env)) return strtoull(e, nullptr, 10) << 20;
  size_t free_b = 0, total_b = 0;
  if (cudaMemGetInfo(&free_b, &total_b) != cudaSuccess) return (size_t)4096 << 20;
  const size_t headroom = (size_t)1 << 30;
  size_t avail = free_b + held > headroom ? free_b + held - headroom : 0;
  return std::min((size_t)(share * (double)total_b), avail);
}

// Block-walk workspace of selection and the fallback: every CTA gets room
// for one whole chart of a row (4,096 columns, 640 n entries, as the
// per-sequence forward charts; EPIC_ENTRIES_PER_CTA overrides), and as many
// CTAs as asked run if their workspaces fit EPIC_WORKSPACE_MB (default a
// quarter of the GPU), else fewer (the kernels loop over their sequences).
epic_status ensure_workspace(epic_lexer_table* t, int want_ctas, int n, cudaStream_t st) {
  const epic_grammar* g = t->g;
  int W = g->dg.W, VW = g->dg.VW, FW = g->dg.FW;
  WsDims d;
  d.nmax = kMaxCols;
  d.emax = std::max<long long>(4096, 640ll * std::max(1, n));
  if (const char* e = getenv("EPIC_ENTRIES_PER_CTA")) d.emax = std::max<long long>(64, atoll(e));
  const size_t budget = workspace_budget("EPIC_WORKSPACE_MB", 0.25, t->d_ws ? t->ws_bytes : 0);
  size_t per = ws_bytes_per_cta(d, W, VW, FW);
  while (per > budget && d.emax > 4096) {  // not even one CTA fits: smaller charts
    d.emax = d.emax * 3 / 4;
    per = ws_bytes_per_cta(d, W, VW, FW);
  }
  int ctas = (int)std::max<long long>(1, std::min<long long>(std::max(1, want_ctas), (long long)(budget / per)));
  size_t need = per * (size_t)ctas;
  if (t->d_ws && t->ws_bytes >= need && t->dims.nmax == d.nmax && t->dims.emax == d.emax) {
    t->ctas = ctas;
    return EPIC_OK;
  }
  if (t->d_ws) {
    cudaStreamSynchronize(t->last);
    cudaFree(t->d_ws);
    t->d_ws = nullptr;
  }
  if (cudaMalloc(&t->d_ws, need) != cudaSuccess) {
    t->d_ws = nullptr;
    return EPIC_ERR_OOM;
  }
  // staging rows and bdone must start at zero; the rest is written before read
  if (cudaMemsetAsync(t->d_ws, 0, need, st) != cudaSuccess) return EPIC_ERR_CUDA;
  t->ws_bytes = need;
  t->dims = d;
  t->ctas = ctas;
  return EPIC_OK;
}

// Warp-walk workspace: columns <= min(4096, 8 n + 256) per walk; entries
// per walk EPIC_ENTRIES_PER_WALK (default 256 n); warps cut down until the
// total fits EPIC_WARP_WORKSPACE_MB (default a quarter of the GPU).
epic_status ensure_wworkspace(epic_lexer_table* t, long long checks, int n, cudaStream_t st) {
  const epic_grammar* g = t->g;
  int W = g->dg.W, VW = g->dg.VW;
  int nmax = std::min(kWCols, 8 * n + 256);
  long long emax = 256ll * std::max(1, n);
  if (const char* e = getenv("EPIC_ENTRIES_PER_WALK")) emax = atoll(e);
  const size_t budget = workspace_budget("EPIC_WARP_WORKSPACE_MB", 0.25, t->d_wws ? t->wws_bytes : 0);
  size_t per = wbytes_per_warp(nmax, emax, W, VW);
  long long warps = std::min<long long>(checks, (long long)sm_count() * 2 * kWarpsPerCta);
  warps = std::max<long long>(kWarpsPerCta, (warps + kWarpsPerCta - 1) / kWarpsPerCta * kWarpsPerCta);
  while (warps > kWarpsPerCta && per * (size_t)warps > budget) warps -= kWarpsPerCta;
  size_t need = per * (size_t)warps;
  if (t->d_wws && t->wws_bytes >= need && t->wnmax == nmax && t->wemax == emax) {
    t->wwarps = (int)std::min<long long>(warps, t->wws_bytes / per / kWarpsPerCta * kWarpsPerCta);
    return EPIC_OK;
  }
  if (t->d_wws) {
    cudaStreamSynchronize(t->last);
    cudaFree(t->d_wws);
    t->d_wws = nullptr;
  }
  if (cudaMalloc(&t->d_wws, need) != cudaSuccess) {
    t->d_wws = nullptr;
    return EPIC_ERR_OOM;
  }
  if (cudaMemsetAsync(t->d_wws, 0, need, st) != cudaSuccess) return EPIC_ERR_CUDA;
  t->wws_bytes = need;
  t->wnmax = nmax;
  t->wemax = emax;
  t->wwarps = (int)warps;
  return EPIC_OK;
}

WPack wpack_of(const epic_lexer_table* t) {
  WPack p;
  p.base = t->d_wws;
  p.nmax = t->wnmax;
  p.emax = t->wemax;
  p.W = t->g->dg.W;
  p.VW = t->g->dg.VW;
  p.per_warp = wbytes_per_warp(p.nmax, p.emax, p.W, p.VW);
  return p;
}

// Grow a device buffer owned by the table (synchronizing its last stream first).
epic_status grow(epic_lexer_table* t, char** buf, size_t* have, size_t need) {
  if (*buf && *have >= need) return EPIC_OK;
  if (*buf) {
    cudaStreamSynchronize(t->last);
    cudaFree(*buf);
    *buf = nullptr;
    *have = 0;
  }
  if (cudaMalloc(buf, need) != cudaSuccess) {
    *buf = nullptr;
    return EPIC_ERR_OOM;
  }
  *have = need;
  return EPIC_OK;
}

// Checks by region, steps 1-2 (also the start of witness extraction): the
// per-sequence arena (EPIC_SEQ_ENTRIES, default 640 n chart entries per
// sequence; EPIC_SEQ_WORKSPACE_MB, default 30 % of the GPU, caps the batch:
// a sequence whose chart does not fit its arena has its checks walk the
// whole graph instead), the forward charts and the good masks with their
// indexes.
epic_status region_prepare(const epic_grammar* g, epic_lexer_table* t, const int32_t* d_x, int B, int n, SeqPack& sp,
                           cudaStream_t st) {
  (void)g;
  const DevGrammar& dg = t->dgl;
  sp.nmax = std::min(kMaxCols, 8 * n + 256);
  sp.n = n;
  sp.W = dg.W;
  sp.VW = dg.VW;
  sp.edge_cap = 32 * sp.nmax;
  sp.emax = 640ll * n;
  if (const char* e = getenv("EPIC_SEQ_ENTRIES")) sp.emax = atoll(e);
  const size_t budget = workspace_budget("EPIC_SEQ_WORKSPACE_MB", 0.30, t->d_seq ? t->seq_bytes : 0);
  while (sp.emax > 4096 && sp.bytes() * (size_t)B > budget) sp.emax = sp.emax * 3 / 4;
  sp.per_seq = sp.bytes();
  epic_status s = grow(t, &t->d_seq, &t->seq_bytes, sp.per_seq * (size_t)B);
  if (s != EPIC_OK) return s;
  sp.base = t->d_seq;
  t->last = st;
  const size_t smem_cap = 190 * 1024;
  const int rmax = 256;
  bool sm = dg.W <= 32;
  // 1. forward charts
  {
    int wpc = kWarpsPerCta;
    size_t per = smem_per_warp(sp.nmax, rmax, dg.W, dg.VW);
    if (sm) wpc = (int)std::min<size_t>(kWarpsPerCta, smem_cap / per);
    // wide item sets: one CTA per sequence (Gauss-Seidel columns); narrow
    // ones: one warp per sequence.  EPIC_FORWARD_CTA=0/1 overrides.
    bool cta_walk = dg.W > 32;
    if (const char* e = getenv("EPIC_FORWARD_CTA")) cta_walk = atoi(e) != 0;
    t->nk = 3;
    t->kname[0] = cta_walk ? "k_forward_gs" : "k_forward";
    t->kname[1] = "k_good";
    t->kname[2] = "k_check";
    mark(t, 0, st);
    if (cta_walk) {
      launch_forward_gs(std::min(B, 4 * sm_count()), st, dg, t->d_table, t->vocab, d_x, B, n, sp, t->d_stats);
    } else if (sm && wpc >= 1) {
      size_t dyn = per * wpc;
      launch_forward(true, (B + wpc - 1) / wpc, 32 * wpc, dyn, st, dg, t->d_table, t->vocab, d_x, B, n, sp, rmax,
                     t->d_stats);
    } else {
      launch_forward(false, (B + kWarpsPerCta - 1) / kWarpsPerCta, 32 * kWarpsPerCta, 0, st, dg, t->d_table,
                     t->vocab, d_x, B, n, sp, 0, t->d_stats);
    }
  }
  // 2. good masks
  mark(t, 1, st);
  launch_good(B, st, dg, B, sp);
  mark(t, 2, st);
  return cudaGetLastError() == cudaSuccess ? EPIC_OK : EPIC_ERR_CUDA;
}

epic_status validate_region(const epic_grammar* g, epic_lexer_table* t, const int32_t* d_x, int B, int n,
                            const int32_t* d_pos, int k, const int32_t* d_cand, int K, uint8_t* d_valid,
                            cudaStream_t st) {
  const DevGrammar& dg = t->dgl;
  long long total = (long long)B * k * K;
  // per-warp workspace of the checks: own columns after the chart's
  WPack wp;
  wp.nmax = kWCols;
  // own entries: the region's columns and the rows carried after it
  wp.emax = std::max(8192ll, 64ll * n);
  if (const char* e = getenv("EPIC_ENTRIES_PER_WALK")) wp.emax = atoll(e);
  wp.W = dg.W;
  wp.VW = dg.VW;
  wp.per_warp = wbytes_per_warp(wp.nmax, wp.emax, wp.W, wp.VW);
  const size_t wbudget = workspace_budget("EPIC_WARP_WORKSPACE_MB", 0.25, t->d_wws ? t->wws_bytes : 0);
  long long warps = std::min<long long>(total, (long long)sm_count() * 2 * kWarpsPerCta);
  warps = std::max<long long>(1, warps);
  warps = std::max<long long>(1, std::min<long long>(warps, (long long)(wbudget / wp.per_warp)));
  size_t wneed = wp.per_warp * (size_t)warps;
  if (!t->d_wws || t->wws_bytes < wneed || t->wnmax != wp.nmax || t->wemax != wp.emax) {
    if (t->d_wws) {
      cudaStreamSynchronize(t->last);
      cudaFree(t->d_wws);
      t->d_wws = nullptr;
    }
    if (cudaMalloc(&t->d_wws, wneed) != cudaSuccess) {
      t->d_wws = nullptr;
      return EPIC_ERR_OOM;
    }
    // the global stage starts at zero; walks return it zeroed
    if (cudaMemsetAsync(t->d_wws, 0, wneed, st) != cudaSuccess) return EPIC_ERR_CUDA;
    t->wws_bytes = wneed;
    t->wnmax = wp.nmax;
    t->wemax = wp.emax;
  }
  wp.base = t->d_wws;
  epic_status s = grow(t, (char**)&t->d_regs, &t->regs_bytes, (size_t)warps * 3 * wp.nmax * 4);
  if (s != EPIC_OK) return s;
  t->last = st;
  const size_t smem_cap = 190 * 1024;
  const int rmax = 256;
  bool sm = dg.W <= 32;
  // 1-2. forward charts and good masks
  SeqPack sp;
  s = region_prepare(g, t, d_x, B, n, sp, st);
  if (s != EPIC_OK) return s;
  t->n_region += total;
  t->n_vkernels += 3;
  // 3. checks
  cudaMemsetAsync(t->d_counter, 0, 8, st);
  size_t per = smem_per_warp(wp.nmax, rmax, dg.W, dg.VW);
  int wpc = sm ? (int)std::min<size_t>(kWarpsPerCta, smem_cap / per) : 0;
  wpc = (int)std::min<long long>(wpc, warps);  // every launched warp owns an allocated workspace
  if (wpc >= 1) {
    int blocks = (int)std::max<long long>(1, warps / wpc);
    size_t dyn = per * wpc;
    launch_check_sm(blocks, 32 * wpc, dyn, st, dg, t->d_table, t->vocab, d_x, n, d_pos, k, d_cand, K, total, d_valid,
                    sp, wp, t->d_regs, rmax, t->d_counter, t->d_stats);
  } else {
    int per_cta = (int)std::min<long long>(kWarpsPerCta, warps);
    int blocks = (int)std::max<long long>(1, warps / per_cta);
    launch_check_global(blocks, 32 * per_cta, 0, st, dg, t->d_table, t->vocab, d_x, n, d_pos, k, d_cand, K, total,
                        d_valid, sp, wp, t->d_regs, 0, t->d_counter, t->d_stats);
  }
  mark(t, 3, st);
  return cudaGetLastError() == cudaSuccess ? EPIC_OK : EPIC_ERR_CUDA;
}

WsPack pack_of(const epic_lexer_table* t) {
  WsPack p;
  p.base = t->d_ws;
  p.dims = t->dims;
  p.W = t->g->dg.W;
  p.VW = t->g->dg.VW;
  p.FW = t->g->dg.FW;
  p.per_cta = ws_bytes_per_cta(t->dims, p.W, p.VW, p.FW);
  return p;
}

}  // namespace

extern "C" {

#ifdef EPIC_PHASE_TIMERS
// measurement build only: per-phase cycle counters (the walks' and the GS
// columns' in out16, the good pass's in out16 + 16)
int epic_debug_phase_read(unsigned long long* out16, int reset) {
  if (cudaDeviceSynchronize() != cudaSuccess) return -1;
  for (int i = 0; i < 16; ++i) out16[i] = 0;
  if (phase_read_walk(out16, reset) != 0 || phase_read_forward(out16, reset) != 0 ||
      phase_read_check_sm(out16, reset) != 0 || phase_read_check_global(out16, reset) != 0)
    return -1;
  for (int i = 0; i < 16; ++i) out16[16 + i] = 0;
  if (phase_read_good(out16 + 16, reset) != 0) return -1;
  return 0;
}
#endif

const char* epic_status_string(epic_status s) {
  switch (s) {
    case EPIC_OK: return "ok";
    case EPIC_ERR_INVALID_ARG: return "invalid argument";
    case EPIC_ERR_GRAMMAR: return "invalid grammar (malformed or empty language)";
    case EPIC_ERR_LEXER: return "invalid lexer specification";
    case EPIC_ERR_OOM: return "out of memory";
    case EPIC_ERR_CUDA: return "CUDA error";
    case EPIC_ERR_CAPACITY: return "capacity exceeded";
    case EPIC_ERR_TIMEOUT: return "device loop bound exceeded";
  }
  return "unknown status";
}

epic_status epic_grammar_create(const epic_grammar_desc* desc, epic_grammar** out) {
  if (!desc || !out) return EPIC_ERR_INVALID_ARG;
  *out = nullptr;
  if (desc->n_terminals <= 0 || desc->n_terminals > 255 || desc->n_nonterminals <= 0 ||
      desc->n_nonterminals > 32 * kMaxVW || desc->n_productions < 0 || !desc->terminal_regex ||
      !desc->terminal_skip || (desc->n_productions > 0 && (!desc->lhs || !desc->rhs_off)))
    return EPIC_ERR_INVALID_ARG;
  int dev_count = 0;
  if (cudaGetDeviceCount(&dev_count) != cudaSuccess || dev_count == 0) return EPIC_ERR_CUDA;
  epic_grammar* g = new (std::nothrow) epic_grammar();
  if (!g) return EPIC_ERR_OOM;
  cudaGetDevice(&g->device);
  int T = desc->n_terminals, V = desc->n_nonterminals, P = desc->n_productions;
  try {
    std::vector<std::string> rx;
    for (int t = 0; t < T; ++t) {
      if (!desc->terminal_regex[t]) throw std::invalid_argument("null regex");
      rx.emplace_back(desc->terminal_regex[t]);
    }
    try {
      g->dfa = build_lexer(rx);
    } catch (std::runtime_error&) {
      delete g;
      return EPIC_ERR_LEXER;
    }
    if (g->dfa.Q > kMaxQ) {
      delete g;
      return EPIC_ERR_CAPACITY;
    }
    std::vector<uint8_t> skip(desc->terminal_skip, desc->terminal_skip + T);
    std::vector<int32_t> lhs(desc->lhs, desc->lhs + P);
    std::vector<int32_t> off(desc->rhs_off, desc->rhs_off + P + 1);
    if (off[0] != 0) throw std::invalid_argument("rhs_off[0] != 0");
    std::vector<int32_t> rhs;
    if (off[P] > 0) {
      if (!desc->rhs) throw std::invalid_argument("null rhs");
      rhs.assign(desc->rhs, desc->rhs + off[P]);
    }
    try {
      g->tabs = build_tables(T, skip, V, desc->start, lhs, off, rhs);
    } catch (std::domain_error&) {
      delete g;
      return EPIC_ERR_GRAMMAR;
    }
  } catch (std::exception&) {
    delete g;
    return EPIC_ERR_INVALID_ARG;
  }
  GrammarTables& G = g->tabs;
  if (G.W > kMaxW) {
    delete g;
    return EPIC_ERR_CAPACITY;
  }
  g->cov = build_cover(G);
  if (g->cov.FW > kMaxFW) {
    delete g;
    return EPIC_ERR_CAPACITY;
  }
  DevGrammar& d = g->dg;
  d.T = G.T;
  d.V = G.V;
  d.D = G.D;
  d.W = G.W;
  d.VW = (G.V + 31) / 32;
  d.Q = g->dfa.Q;
  d.start_item = G.start_item;
  d.accept_item = G.accept_item;
  std::vector<uint32_t> next_any(G.W);
  for (int w = 0; w < G.W; ++w) next_any[w] = G.any_term[w] | G.any_nt[w];
  std::vector<int16_t> inext(G.D), ilhs(G.D);
  for (int i = 0; i < G.D; ++i) {
    inext[i] = (int16_t)G.item_next[i];
    ilhs[i] = (int16_t)G.item_lhs[i];
  }
  epic_status st = EPIC_OK;
  auto up = [&](auto& v, auto** o) {
    if (st == EPIC_OK) st = upload(g, v, o);
  };
  up(G.exp_term, &d.exp_term);
  up(G.exp_nt, &d.exp_nt);
  up(G.any_nt, &d.any_nt);
  up(G.any_term, &d.any_term);
  up(next_any, &d.next_any);
  up(G.nullable_next, &d.nullable_next);
  up(G.complete, &d.complete);
  up(G.pred, &d.pred);
  up(G.gap_pred, &d.gap_pred);
  up(inext, &d.item_next);
  up(ilhs, &d.item_lhs);
  up(g->dfa.accept, &d.dfa_accept);
  up(g->dfa.next, &d.dfa_next);
  std::vector<uint8_t> ext(g->dfa.Q, 0);
  for (int q = 0; q < g->dfa.Q; ++q)
    for (int c = 0; c < 256; ++c)
      if (g->dfa.next[(size_t)q * 256 + c] >= 0) ext[q] = 1;
  up(ext, &d.dfa_ext);
  up(G.skip, &d.skip);
  {
    // runs of advanceable items for the doubling closure (see device.cuh)
    int maxlen = 0;
    for (size_t p = 0; p + 1 < G.rhs_off.size(); ++p) maxlen = std::max(maxlen, G.rhs_off[p + 1] - G.rhs_off[p]);
    int steps = 1;
    while ((1 << steps) <= maxlen) ++steps;
    d.adv_steps = steps;
    std::vector<uint32_t> pw((size_t)2 * steps * G.W, 0);
    auto bit = [&](const std::vector<uint32_t>& m, long long i) -> bool {
      return i >= 0 && i < (long long)G.W * 32 && ((m[(size_t)(i >> 5)] >> (i & 31)) & 1u);
    };
    for (int mode = 0; mode < 2; ++mode) {
      std::vector<uint32_t> cur = mode ? next_any : G.nullable_next;
      for (int st2 = 0; st2 < steps; ++st2) {
        std::copy(cur.begin(), cur.end(), pw.begin() + ((size_t)mode * steps + st2) * G.W);
        const long long k = 1ll << st2;  // next: i and i + k both start runs of length k
        std::vector<uint32_t> nx(G.W, 0);
        for (long long i = 0; i < (long long)G.W * 32; ++i)
          if (bit(cur, i) && bit(cur, i + k)) nx[(size_t)(i >> 5)] |= 1u << (i & 31);
        cur.swap(nx);
      }
    }
    up(pw, &d.adv_pow);
  }
  {
    // witness extraction tables: complete items by left side, and a shortest
    // terminal string of every nonterminal (fixpoint of the shortest yield
    // length; a production is chosen only when it strictly shortens, so the
    // choices form no cycle and expand to finite strings)
    const int V = G.V, T = G.T;
    const int P2 = (int)G.lhs.size();
    std::vector<int32_t> coff(V + 1, 0), citems;
    for (int p = 0; p < P2; ++p)
      if (G.lhs[p] >= 0) ++coff[G.lhs[p] + 1];
    for (int v = 0; v < V; ++v) coff[v + 1] += coff[v];
    citems.assign(coff[V], 0);
    std::vector<int32_t> cur(coff.begin(), coff.end() - 1);
    for (int p = 0; p < P2; ++p)
      if (G.lhs[p] >= 0) citems[cur[G.lhs[p]]++] = G.item_base[p] + (G.rhs_off[p + 1] - G.rhs_off[p]);
    const long long INF = 1ll << 40;
    std::vector<long long> len(V, INF);
    std::vector<int> best(V, -1);
    for (bool changed = true; changed;) {
      changed = false;
      for (int p = 0; p < P2; ++p) {
        if (G.lhs[p] < 0) continue;
        long long L = 0;
        for (int i = G.rhs_off[p]; i < G.rhs_off[p + 1] && L < INF; ++i) {
          const int X = G.rhs[i];
          L += X < T ? 1 : len[X - T];
        }
        if (L < len[G.lhs[p]]) {
          len[G.lhs[p]] = L;
          best[G.lhs[p]] = p;
          changed = true;
        }
      }
    }
    std::vector<int32_t> yoff(V + 1, 0), ys;
    std::vector<std::vector<int32_t>> memo(V);
    std::vector<char> done(V, 0);
    std::function<void(int, std::vector<int32_t>&)> expand = [&](int A, std::vector<int32_t>& out) {
      if (done[A]) {
        out.insert(out.end(), memo[A].begin(), memo[A].end());
        return;
      }
      std::vector<int32_t> mine;
      const int p = best[A];
      if (p >= 0 && mine.size() < 4096)
        for (int i = G.rhs_off[p]; i < G.rhs_off[p + 1]; ++i) {
          const int X = G.rhs[i];
          if (X < T) mine.push_back(X);
          else expand(X - T, mine);
        }
      if (mine.size() > 4096) mine.resize(4096);
      memo[A] = mine;
      done[A] = 1;
      out.insert(out.end(), mine.begin(), mine.end());
    };
    for (int v = 0; v < V; ++v) {
      std::vector<int32_t> y;
      if (len[v] < INF) expand(v, y);
      yoff[v + 1] = yoff[v] + (int)y.size();
      ys.insert(ys.end(), y.begin(), y.end());
    }
    up(coff, &d.nt_comp_off);
    up(citems, &d.nt_comp);
    up(yoff, &d.ny_off);
    up(ys, &d.ny);
  }
  d.FS = g->cov.FS;
  d.FW = g->cov.FW;
  d.cov_start = g->cov.start;
  d.cov_accept = g->cov.accept;
  up(g->cov.eps_close, &d.cov_eps_close);
  up(g->cov.all_close, &d.cov_all_close);
  if (st != EPIC_OK) {
    epic_grammar_destroy(g);
    return st;
  }
  *out = g;
  return EPIC_OK;
}

void epic_grammar_destroy(epic_grammar* g) {
  if (!g) return;
  for (void* p : g->dev_allocs) cudaFree(p);
  delete g;
}

int32_t epic_grammar_lexer_states(const epic_grammar* g) { return g ? g->dfa.Q : -1; }

epic_status epic_lexer_table_build(const epic_grammar* g, const int32_t* tok_off, const uint8_t* tok_bytes,
                                   int32_t vocab, void* cuda_stream, epic_lexer_table** out) {
  if (!g || !tok_off || !out || vocab <= 0) return EPIC_ERR_INVALID_ARG;
  *out = nullptr;
  if (tok_off[0] != 0) return EPIC_ERR_INVALID_ARG;
  for (int t = 0; t < vocab; ++t) {
    int L = tok_off[t + 1] - tok_off[t];
    if (L < 1 || L > 64) return EPIC_ERR_INVALID_ARG;
  }
  if (!tok_bytes) return EPIC_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  epic_lexer_table* t = new (std::nothrow) epic_lexer_table();
  if (!t) return EPIC_ERR_OOM;
  t->g = g;
  t->vocab = vocab;
  t->last = st;
  t->dgl = g->dg;
  t->dgl.lazy = LazyLex{};
  int Q = g->dg.Q;
  size_t nbytes = (size_t)tok_off[vocab];
  int32_t* d_off = nullptr;
  uint8_t* d_bytes = nullptr;
  int* d_ovf = nullptr;
  epic_status res = EPIC_OK;
  if (cudaMalloc(&t->d_table, (size_t)vocab * Q * sizeof(LexEntry)) != cudaSuccess ||
      cudaMalloc(&d_off, (size_t)(vocab + 1) * 4) != cudaSuccess || cudaMalloc(&d_bytes, nbytes) != cudaSuccess ||
      cudaMalloc(&d_ovf, 4) != cudaSuccess || cudaMalloc(&t->d_stats, S_N * 8) != cudaSuccess ||
      cudaMalloc(&t->d_counter, 8) != cudaSuccess) {
    res = EPIC_ERR_OOM;
  }
  if (res == EPIC_OK) {
    cudaMemcpyAsync(d_off, tok_off, (size_t)(vocab + 1) * 4, cudaMemcpyHostToDevice, st);
    cudaMemcpyAsync(d_bytes, tok_bytes, nbytes, cudaMemcpyHostToDevice, st);
    cudaMemsetAsync(d_ovf, 0, 4, st);
    cudaMemsetAsync(t->d_stats, 0, S_N * 8, st);
    long long total = (long long)vocab * Q;
    int threads = 256;
    long long blocks = (total + threads - 1) / threads;
    k_lex_table<<<(unsigned)blocks, threads, 0, st>>>(d_off, d_bytes, vocab, Q, g->dg.dfa_next, g->dg.dfa_accept,
                                                       g->dg.skip, t->d_table, d_ovf);
    int ovf = 0;
    if (cudaGetLastError() != cudaSuccess || cudaMemcpyAsync(&ovf, d_ovf, 4, cudaMemcpyDeviceToHost, st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess)
      res = EPIC_ERR_CUDA;
    else if (ovf)
      res = EPIC_ERR_CAPACITY;
  }
  cudaFree(d_off);
  cudaFree(d_bytes);
  cudaFree(d_ovf);
  if (res != EPIC_OK) {
    epic_lexer_table_destroy(t);
    return res;
  }
  t->dgl.lazy.stats = t->d_stats + S_LEX_LOOKUPS;  // lookups are counted for dense tables too
  *out = t;
  return EPIC_OK;
}

epic_status epic_lexer_table_build_lazy(const epic_grammar* g, const int32_t* tok_off, const uint8_t* tok_bytes,
                                        int32_t vocab, int64_t capacity, void* cuda_stream, epic_lexer_table** out) {
  if (!g || !tok_off || !out || vocab <= 0 || capacity < 1) return EPIC_ERR_INVALID_ARG;
  *out = nullptr;
  if (tok_off[0] != 0) return EPIC_ERR_INVALID_ARG;
  for (int t = 0; t < vocab; ++t) {
    int L = tok_off[t + 1] - tok_off[t];
    if (L < 1 || L > 64) return EPIC_ERR_INVALID_ARG;
  }
  if (!tok_bytes) return EPIC_ERR_INVALID_ARG;
  // the key token * Q + state + 1 must fit 32 bits
  if ((unsigned long long)vocab * (unsigned long long)g->dg.Q >= 0xFFFFFFFFull) return EPIC_ERR_CAPACITY;
  long long cap = 1;
  while (cap < capacity) cap <<= 1;
  if (cap > (1ll << 30)) return EPIC_ERR_CAPACITY;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  epic_lexer_table* t = new (std::nothrow) epic_lexer_table();
  if (!t) return EPIC_ERR_OOM;
  t->g = g;
  t->vocab = vocab;
  t->last = st;
  t->lz_cap = cap;
  size_t nbytes = (size_t)tok_off[vocab];
  epic_status res = EPIC_OK;
  if (cudaMalloc(&t->d_lz_keys, (size_t)cap * 4) != cudaSuccess ||
      cudaMalloc(&t->d_lz_ready, (size_t)cap * 4) != cudaSuccess ||
      cudaMalloc(&t->d_lz_vals, (size_t)cap * sizeof(LexEntry)) != cudaSuccess ||
      cudaMalloc(&t->d_lz_off, (size_t)(vocab + 1) * 4) != cudaSuccess ||
      cudaMalloc(&t->d_lz_bytes, nbytes) != cudaSuccess || cudaMalloc(&t->d_stats, S_N * 8) != cudaSuccess ||
      cudaMalloc(&t->d_counter, 8) != cudaSuccess)
    res = EPIC_ERR_OOM;
  if (res == EPIC_OK) {
    cudaMemcpyAsync(t->d_lz_off, tok_off, (size_t)(vocab + 1) * 4, cudaMemcpyHostToDevice, st);
    cudaMemcpyAsync(t->d_lz_bytes, tok_bytes, nbytes, cudaMemcpyHostToDevice, st);
    cudaMemsetAsync(t->d_lz_keys, 0, (size_t)cap * 4, st);
    cudaMemsetAsync(t->d_lz_ready, 0, (size_t)cap * 4, st);
    cudaMemsetAsync(t->d_stats, 0, S_N * 8, st);
    if (cudaGetLastError() != cudaSuccess || cudaStreamSynchronize(st) != cudaSuccess) res = EPIC_ERR_CUDA;
  }
  if (res != EPIC_OK) {
    epic_lexer_table_destroy(t);
    return res;
  }
  t->dgl = g->dg;
  t->dgl.lazy.keys = t->d_lz_keys;
  t->dgl.lazy.ready = t->d_lz_ready;
  t->dgl.lazy.vals = t->d_lz_vals;
  t->dgl.lazy.mask = (uint32_t)(cap - 1);
  t->dgl.lazy.tok_off = t->d_lz_off;
  t->dgl.lazy.tok_bytes = t->d_lz_bytes;
  t->dgl.lazy.stats = t->d_stats + S_LEX_LOOKUPS;
  *out = t;
  return EPIC_OK;
}

void epic_lexer_table_destroy(epic_lexer_table* t) {
  if (!t) return;
  if (t->last) cudaStreamSynchronize(t->last);
  cudaFree(t->d_table);
  cudaFree(t->d_ws);
  cudaFree(t->d_wws);
  cudaFree(t->d_spec);
  cudaFree(t->d_seq);
  cudaFree(t->d_regs);
  cudaFree(t->d_wit);
  cudaFree(t->d_fb);
  cudaFree(t->d_stats);
  cudaFree(t->d_counter);
  cudaFree(t->d_lz_keys);
  cudaFree(t->d_lz_ready);
  cudaFree(t->d_lz_vals);
  cudaFree(t->d_lz_off);
  cudaFree(t->d_lz_bytes);
  for (cudaEvent_t e : t->kev)
    if (e) cudaEventDestroy(e);
  for (cudaEvent_t e : t->sev)
    if (e) cudaEventDestroy(e);
  delete t;
}

epic_status epic_lexer_table_copy(const epic_lexer_table* t, int32_t first_token, int32_t count, void* host_out,
                                  size_t out_bytes) {
  if (!t || !host_out || first_token < 0 || count < 0 || first_token + count > t->vocab || !t->d_table)
    return EPIC_ERR_INVALID_ARG;
  size_t Q = (size_t)t->g->dg.Q;
  size_t bytes = (size_t)count * Q * sizeof(LexEntry);
  if (out_bytes < bytes) return EPIC_ERR_INVALID_ARG;
  if (cudaStreamSynchronize(t->last) != cudaSuccess) return EPIC_ERR_CUDA;
  if (cudaMemcpy(host_out, t->d_table + (size_t)first_token * Q, bytes, cudaMemcpyDeviceToHost) != cudaSuccess)
    return EPIC_ERR_CUDA;
  return EPIC_OK;
}

epic_status epic_validate_batch(const epic_grammar* g, const epic_lexer_table* tc, const int32_t* d_x, int32_t B,
                                int32_t n, const int32_t* d_pos, int32_t k, const int32_t* d_cand, int32_t K,
                                uint8_t* d_valid, void* cuda_stream) {
  epic_lexer_table* t = const_cast<epic_lexer_table*>(tc);
  if (!g || !t || t->g != g || B < 0 || n < 0 || k < 0 || K < 0) return EPIC_ERR_INVALID_ARG;
  long long total = (long long)B * k * K;
  if (total == 0) return EPIC_OK;
  if (!d_x || !d_pos || !d_cand || !d_valid || n == 0) return EPIC_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  // Checks by region over a per-sequence chart when the item sets are wide
  // (whole-graph walks of large grammars are far too long) or when there are
  // more checks than resident walks: the chart of x is then built once per
  // sequence instead of once per check.
  bool region = g->dg.W > 32 || total > (long long)sm_count() * 2 * kWarpsPerCta;
  if (const char* e = getenv("EPIC_REGION")) region = atoi(e) != 0;
  if (region) return validate_region(g, t, d_x, B, n, d_pos, k, d_cand, K, d_valid, st);
  epic_status s = ensure_wworkspace(t, total, n, st);
  if (s != EPIC_OK) return s;
  t->last = st;
  cudaMemsetAsync(t->d_counter, 0, 8, st);
  // rows of the open column in shared memory (512 slots per warp, as many
  // warps per CTA as fit) when the item set is narrow, else the global stage
  WPack wp = wpack_of(t);
  const size_t smem_cap = 190 * 1024;  // + 27 KB static per CTA <= 227 KB
  const int rmax = 256;
  size_t per = smem_per_warp(wp.nmax, rmax, wp.W, wp.VW);
  const DevGrammar& dg = t->dgl;
  size_t gt = gtab_bytes(dg.T, dg.V, dg.W, dg.D, dg.Q);
  int gsm = (gt + 4 * per <= smem_cap) ? 1 : 0;  // tables in shared memory if 4 warps still fit
  int wpc = (int)std::min<size_t>(kWarpsPerCta, (smem_cap - (gsm ? gt : 0)) / per);
  if (const char* e = getenv("EPIC_GLOBAL_STAGE"))
    if (atoi(e)) wpc = 0;
  if (wp.W > 32) wpc = 0;
  // spread the walks over every SM: no more warps per CTA than walks per SM
  int per_sm = (int)((t->wwarps + sm_count() - 1) / sm_count());
  if (wpc > per_sm) wpc = std::max(2, per_sm);
  t->n_vkernels += 1;
  t->nk = 1;
  t->kname[0] = "k_validate_warp";
  mark(t, 0, st);
  if (wpc >= 2) {
    size_t dyn = per * wpc + (gsm ? gt : 0);
    int blocks = (t->wwarps + wpc - 1) / wpc;
    if ((size_t)blocks * wpc > (size_t)t->wwarps) blocks = t->wwarps / wpc;
    launch_validate_warp(true, blocks, 32 * wpc, dyn, st, t->dgl, t->d_table, t->vocab, d_x, n, d_pos, k, d_cand, K,
                         total, d_valid, wp, rmax, gsm, t->d_counter, t->d_stats);
  } else {
    launch_validate_warp(false, t->wwarps / kWarpsPerCta, 32 * kWarpsPerCta, 0, st, t->dgl, t->d_table, t->vocab, d_x,
                         n, d_pos, k, d_cand, K, total, d_valid, wp, 0, 0, t->d_counter, t->d_stats);
  }
  mark(t, 1, st);
  return cudaGetLastError() == cudaSuccess ? EPIC_OK : EPIC_ERR_CUDA;
}

int epic_last_kernel_times(const epic_lexer_table* t, float* ms, const char** names, int cap) {
  if (!t || (!ms && cap > 0) || cap < 0) return -1;
  int n = 0;
  if (t->nk > 0) {
    for (int i = 0; i <= t->nk; ++i)
      if (!t->kev[i]) return -1;
    if (cudaEventSynchronize(t->kev[t->nk]) != cudaSuccess) return -1;
    for (int i = 0; i < t->nk && n < cap; ++i, ++n) {
      if (cudaEventElapsedTime(&ms[n], t->kev[i], t->kev[i + 1]) != cudaSuccess) return -1;
      if (names) names[n] = t->kname[i];
    }
  }
  if (t->sel_timed) {
    static const char* sname[2] = {"k_select_spec", "k_select"};
    if (cudaEventSynchronize(t->sev[2]) != cudaSuccess) return -1;
    for (int i = 0; i < 2 && n < cap; ++i, ++n) {
      if (cudaEventElapsedTime(&ms[n], t->sev[i], t->sev[i + 1]) != cudaSuccess) return -1;
      if (names) names[n] = sname[i];
    }
  }
  return n;
}

}  // extern "C"

// ---------------------------------------------------------------- no-alloc validation
// Scratch of epic_validate_batch_noalloc: a fixed device array that every GPU
// which loads this library holds until the process exits.  Its first 256
// bytes hold the work counter; the rest is carved into per-warp workspaces.
constexpr size_t kNoAllocBytes = (size_t)128 << 20;
constexpr int kNoAllocWideMaxN = 128;  // row length limit when item sets exceed 32 words
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

namespace {
std::mutex g_noalloc_mu;
void* g_noalloc_ptr[256] = {nullptr};  // device address of the array, per device ordinal
}  // namespace

extern "C" {

epic_status epic_validate_batch_noalloc(const epic_grammar* g, const epic_lexer_table* tc, const int32_t* d_x,
                                        int32_t B, int32_t n, const int32_t* d_pos, int32_t k,
                                        const int32_t* d_cand, int32_t K, uint8_t* d_valid, void* cuda_stream) {
  epic_lexer_table* t = const_cast<epic_lexer_table*>(tc);
  if (!g || !t || t->g != g || B < 0 || n < 0 || k < 0 || K < 0) return EPIC_ERR_INVALID_ARG;
  long long total = (long long)B * k * K;
  if (total == 0) return EPIC_OK;
  if (!d_x || !d_pos || !d_cand || !d_valid || n == 0) return EPIC_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 256) return EPIC_ERR_CUDA;
  char* base = nullptr;
  {
    // set-up, once per device, with that device current: host code may not
    // use the array's name as a device address
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return EPIC_ERR_CUDA;
      g_noalloc_ptr[dev] = p;
    }
    base = (char*)g_noalloc_ptr[dev];
  }
  const int W = g->dg.W, VW = g->dg.VW;
  // Wide item sets walk the whole graph per check with rows in the global
  // stage, which takes seconds per check on long rows of large grammars; the
  // fixed array holds too few walks for that to finish in reasonable time,
  // so such calls are limited to short rows.
  if (W > 32 && n > kNoAllocWideMaxN) return EPIC_ERR_CAPACITY;
  WPack wp;
  wp.base = base + 256;
  wp.nmax = std::min(kWCols, 8 * n + 256);
  wp.emax = 256ll * n;
  wp.W = W;
  wp.VW = VW;
  wp.per_warp = wbytes_per_warp(wp.nmax, wp.emax, W, VW);
  long long fit = (long long)((kNoAllocBytes - 256) / wp.per_warp);
  if (fit < 1) return EPIC_ERR_CAPACITY;  // one walk's workspace does not fit the array
  const size_t smem_cap = 190 * 1024;
  const int rmax = 256;
  size_t sper = smem_per_warp(wp.nmax, rmax, W, VW);
  int wpc = (W > 32) ? 0 : (int)std::min<size_t>(kWarpsPerCta, smem_cap / sper);
  unsigned long long* counter = (unsigned long long*)base;
  // the kernel reads the table's lex entries and adds into its counters:
  // epic_get_stats and epic_lexer_table_destroy synchronize this stream
  t->last = st;
  if (cudaMemsetAsync(counter, 0, sizeof(unsigned long long), st) != cudaSuccess) return EPIC_ERR_CUDA;
  t->n_vkernels += 1;
  if (wpc >= 2) {
    long long warps = std::min<long long>({total, fit, (long long)sm_count() * 2 * kWarpsPerCta});
    int per_cta = (int)std::min<long long>(wpc, warps);
    int blocks = (int)(warps / per_cta);
    size_t dyn = sper * per_cta;
    launch_validate_warp(true, blocks, 32 * per_cta, dyn, st, t->dgl, t->d_table, t->vocab, d_x, n, d_pos, k, d_cand,
                         K, total, d_valid, wp, rmax, 0, counter, t->d_stats);
  } else {
    // the global stage and its completed-NT sets must start at zero
    long long warps = std::min<long long>({total, fit, (long long)sm_count() * 2 * kWarpsPerCta});
    int per_cta = (int)std::min<long long>(kWarpsPerCta, warps);
    int blocks = (int)(warps / per_cta);
    if (cudaMemsetAsync(wp.base, 0, wp.per_warp * (size_t)blocks * per_cta, st) != cudaSuccess) return EPIC_ERR_CUDA;
    launch_validate_warp(false, blocks, 32 * per_cta, 0, st, t->dgl, t->d_table, t->vocab, d_x, n, d_pos, k, d_cand,
                         K, total, d_valid, wp, 0, 0, counter, t->d_stats);
  }
  return cudaGetLastError() == cudaSuccess ? EPIC_OK : EPIC_ERR_CUDA;
}

epic_status epic_pick_candidates(const int32_t* d_cand, const float* d_cand_conf, const uint8_t* d_valid, int32_t B,
                                 int32_t k, int32_t K, int32_t* d_tok, float* d_conf, void* cuda_stream) {
  if (B < 0 || k < 0 || K < 0) return EPIC_ERR_INVALID_ARG;
  long long total = (long long)B * k;
  if (total == 0) return EPIC_OK;
  if (!d_cand || !d_cand_conf || !d_valid || !d_tok || !d_conf) return EPIC_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  k_pick<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(d_cand, d_cand_conf, d_valid, B, k, K, d_tok, d_conf);
  return cudaGetLastError() == cudaSuccess ? EPIC_OK : EPIC_ERR_CUDA;
}

epic_status epic_select_compatible_subset(const epic_grammar* g, const epic_lexer_table* tc, const int32_t* d_x,
                                          int32_t B, int32_t n, const int32_t* d_pos, int32_t k,
                                          const int32_t* d_tok, const float* d_conf, uint8_t* d_selected,
                                          void* cuda_stream) {
  epic_lexer_table* t = const_cast<epic_lexer_table*>(tc);
  if (!g || !t || t->g != g || B < 0 || n < 0 || k < 0 || k > kMaxSel) return EPIC_ERR_INVALID_ARG;
  if ((long long)B * k == 0) return EPIC_OK;
  if (!d_x || !d_pos || !d_tok || !d_conf || !d_selected || n == 0) return EPIC_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  int want = std::min(2 * B, sm_count() * 2);
  epic_status s = ensure_workspace(t, want, n, st);
  if (s != EPIC_OK) return s;
  if (t->spec_cap < B) {
    if (t->d_spec) {
      cudaStreamSynchronize(t->last);
      cudaFree(t->d_spec);
    }
    t->d_spec = nullptr;
    if (cudaMalloc(&t->d_spec, (size_t)2 * B) != cudaSuccess) return EPIC_ERR_OOM;
    t->spec_cap = B;
  }
  t->last = st;
  mark_event(&t->sev[0], st);
  launch_select_spec(std::min(2 * B, t->ctas), st, t->dgl, t->d_table, t->vocab, d_x, B, n, d_pos, k, d_tok,
                     t->d_spec, pack_of(t));
  mark_event(&t->sev[1], st);
  int ctas = std::min(B, t->ctas);
  launch_select(ctas, st, t->dgl, t->d_table, t->vocab, d_x, B, n, d_pos, k, d_tok, d_conf, d_selected, pack_of(t),
                t->d_spec, t->d_stats);
  mark_event(&t->sev[2], st);
  t->sel_timed = t->sev[0] && t->sev[1] && t->sev[2];
  return cudaGetLastError() == cudaSuccess ? EPIC_OK : EPIC_ERR_CUDA;
}

epic_status epic_fallback_commit(const epic_grammar* g, const epic_lexer_table* tc, int32_t* d_x, int32_t B,
                                 int32_t n, const int32_t* d_pos, int32_t k, const int32_t* d_cand,
                                 const float* d_cand_conf, int32_t K, const int32_t* d_n_target,
                                 const uint8_t* d_selected, const uint8_t* d_valid, int32_t* d_filled,
                                 void* cuda_stream) {
  epic_lexer_table* t = const_cast<epic_lexer_table*>(tc);
  if (!g || !t || t->g != g || B < 0 || n < 0 || k < 0 || K < 0) return EPIC_ERR_INVALID_ARG;
  if ((long long)B * k == 0) return EPIC_OK;
  if ((long long)k * K > kMaxFallbackCand) return EPIC_ERR_CAPACITY;
  if (!d_x || !d_pos || !d_cand || !d_cand_conf || !d_n_target || !d_filled || n == 0 || K == 0)
    return EPIC_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  const int nc = k * K;
  // rounds of m tests per sequence, as many CTAs as two per SM (at most
  // kMaxFallbackSpec tests per sequence, at least one)
  int m = std::max(1, std::min(kMaxFallbackSpec, std::min(nc, (2 * sm_count()) / B)));
  epic_status s = ensure_workspace(t, std::min((long long)B * m, (long long)sm_count() * 2), n, st);
  if (s != EPIC_OK) return s;
  m = std::max(1, std::min(m, t->ctas / B));
  auto r16 = [](size_t b) { return (b + 15) & ~(size_t)15; };
  const size_t o_fb = r16((size_t)B * nc), o_res = o_fb + r16((size_t)B * 2 * 4),
               o_act = o_res + r16((size_t)B * m * 2 * 4), need = o_act + 16;
  s = grow(t, &t->d_fb, &t->fb_bytes, need);
  if (s != EPIC_OK) return s;
  t->last = st;
  uint8_t* rej = (uint8_t*)t->d_fb;
  int32_t* fb = (int32_t*)(t->d_fb + o_fb);
  int32_t* res = (int32_t*)(t->d_fb + o_res);
  unsigned long long* act = (unsigned long long*)(t->d_fb + o_act);
  unsigned long long h_act = 0;
  auto read_active = [&]() -> bool {
    if (cudaMemcpyAsync(&h_act, act, 8, cudaMemcpyDeviceToHost, st) != cudaSuccess) return false;
    return cudaStreamSynchronize(st) == cudaSuccess;
  };
  if (cudaMemsetAsync(act, 0, 8, st) != cudaSuccess) return EPIC_ERR_CUDA;
  launch_fallback_init(B, st, n, d_pos, k, d_cand_conf, K, d_n_target, d_selected, d_valid, d_filled, rej, fb, act,
                       t->d_stats);
  if (!read_active()) return EPIC_ERR_CUDA;
  const int grid = (int)std::min<long long>((long long)B * m, t->ctas);
  for (int round = 0; round <= nc && h_act > 0; ++round) {  // each round rejects or commits a candidate
    launch_fallback_round(grid, st, t->dgl, t->d_table, t->vocab, d_x, B, n, d_pos, k, d_cand, d_cand_conf, K, m, rej,
                          fb, res, pack_of(t), t->d_stats);
    if (cudaMemsetAsync(act, 0, 8, st) != cudaSuccess) return EPIC_ERR_CUDA;
    launch_fallback_resolve(B, st, d_x, n, d_pos, k, d_cand, K, m, rej, fb, res, d_filled, act, t->d_stats);
    ++t->n_fb_rounds;
    if (!read_active()) return EPIC_ERR_CUDA;
  }
  return cudaGetLastError() == cudaSuccess ? EPIC_OK : EPIC_ERR_CUDA;
}

epic_status epic_extract_witness(const epic_grammar* g, const epic_lexer_table* tc, const int32_t* d_x, int32_t B,
                                 int32_t n, int32_t* d_terms, int32_t cap, int32_t* d_len, void* cuda_stream) {
  epic_lexer_table* t = const_cast<epic_lexer_table*>(tc);
  if (!g || !t || t->g != g || B < 0 || n < 0 || cap < 1) return EPIC_ERR_INVALID_ARG;
  if (B == 0) return EPIC_OK;
  if (!d_x || !d_terms || !d_len || n == 0) return EPIC_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  SeqPack sp;
  epic_status s = region_prepare(g, t, d_x, B, n, sp, st);
  if (s != EPIC_OK) return s;
  const size_t per = witness_scratch_bytes(cap, t->dgl.D, t->dgl.W, t->dgl.VW);
  s = grow(t, &t->d_wit, &t->wit_bytes, per * (size_t)B);
  if (s != EPIC_OK) return s;
  launch_witness(B, st, t->dgl, sp, d_terms, cap, d_len, t->d_wit, t->d_stats);
  return cudaGetLastError() == cudaSuccess ? EPIC_OK : EPIC_ERR_CUDA;
}

epic_status epic_commit(int32_t* d_x, int32_t B, int32_t n, const int32_t* d_pos, int32_t k, const int32_t* d_tok,
                        const uint8_t* d_selected, void* cuda_stream) {
  if (B < 0 || n < 0 || k < 0) return EPIC_ERR_INVALID_ARG;
  long long total = (long long)B * k;
  if (total == 0) return EPIC_OK;
  if (!d_x || !d_pos || !d_tok || !d_selected) return EPIC_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  k_commit<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(d_x, B, n, d_pos, k, d_tok, d_selected);
  return cudaGetLastError() == cudaSuccess ? EPIC_OK : EPIC_ERR_CUDA;
}

epic_status epic_get_stats(const epic_lexer_table* t, epic_stats* out, size_t out_bytes, int reset) {
  if (!t || !out || out_bytes < sizeof(epic_stats)) return EPIC_ERR_INVALID_ARG;
  unsigned long long h[S_N];
  if (cudaStreamSynchronize(t->last) != cudaSuccess) return EPIC_ERR_CUDA;
  if (cudaMemcpy(h, t->d_stats, sizeof(h), cudaMemcpyDeviceToHost) != cudaSuccess) return EPIC_ERR_CUDA;
  out->checks = h[S_CHECKS];
  out->valid = h[S_VALID];
  out->overflow = h[S_OVERFLOW];
  out->bad_inputs = h[S_BAD];
  out->columns = h[S_COLUMNS];
  out->entries = h[S_ENTRIES];
  out->cover_checks = h[S_COVER];
  out->exact_checks = h[S_EXACT];
  out->selected = h[S_SELECTED];
  out->lex_lookups = h[S_LEX_LOOKUPS];
  out->lex_misses = h[S_LEX_MISSES];
  out->lex_uncached = h[S_LEX_UNCACHED];
  out->witness_failures = h[S_WITNESS_FAIL];
  out->fallback_rounds = t->n_fb_rounds;
  out->fallback_checks = h[S_FB_CHECKS];
  out->fallback_commits = h[S_FB_COMMITS];
  out->region_checks = t->n_region;
  out->validate_kernels = t->n_vkernels;
  if (reset) {
    if (cudaMemset(t->d_stats, 0, sizeof(h)) != cudaSuccess) return EPIC_ERR_CUDA;
    t->n_region = 0;
    t->n_vkernels = 0;
    t->n_fb_rounds = 0;
  }
  return EPIC_OK;
}

}  // extern "C"
