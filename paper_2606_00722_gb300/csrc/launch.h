// Host-side launchers of the kernels compiled in their own translation units
// (kernels_walk.cu, region_*.cu, kernels_select.cu), so that the
// library's device code builds in parallel.  Each takes the launch shape and
// stream followed by the kernel's own arguments; `sm` selects the variant
// that stages rows in shared memory (its dynamic shared memory is `dyn`).
#pragma once
#include <cuda_runtime.h>

#include "gscols.cuh"
#include "packs.cuh"
#include "seqpack.cuh"

namespace epic {

// whole-graph walks, one warp per check
void launch_validate_warp(bool sm, dim3 grid, dim3 block, size_t dyn, cudaStream_t st, const DevGrammar& g,
                          const LexEntry* table, int vocab, const int32_t* x, int n, const int32_t* pos, int k,
                          const int32_t* cand, int K, long long total, uint8_t* valid, const WPack& wp, int rmax,
                          int gsm, unsigned long long* counter, unsigned long long* stats);

// checks by region
void launch_forward(bool sm, dim3 grid, dim3 block, size_t dyn, cudaStream_t st, const DevGrammar& g,
                    const LexEntry* table, int vocab, const int32_t* x, int B, int n, const SeqPack& sp, int rmax,
                    unsigned long long* stats);
void launch_forward_gs(dim3 grid, cudaStream_t st, const DevGrammar& g, const LexEntry* table, int vocab,
                       const int32_t* x, int B, int n, const SeqPack& sp, unsigned long long* stats);
void launch_good(dim3 grid, cudaStream_t st, const DevGrammar& g, int B, const SeqPack& sp);
void launch_check_sm(dim3 grid, dim3 block, size_t dyn, cudaStream_t st, const DevGrammar& g, const LexEntry* table,
                     int vocab, const int32_t* x, int n, const int32_t* pos, int k, const int32_t* cand, int K,
                     long long total, uint8_t* valid, const SeqPack& sp, const WPack& wp, int32_t* regs, int rmax,
                     unsigned long long* counter, unsigned long long* stats);
void launch_check_global(dim3 grid, dim3 block, size_t dyn, cudaStream_t st, const DevGrammar& g,
                         const LexEntry* table, int vocab, const int32_t* x, int n, const int32_t* pos, int k,
                         const int32_t* cand, int K, long long total, uint8_t* valid, const SeqPack& sp,
                         const WPack& wp, int32_t* regs, int rmax, unsigned long long* counter,
                         unsigned long long* stats);
int good_warps();  // warps per CTA of the good pass

// Alg. 4
void launch_select_spec(dim3 grid, cudaStream_t st, const DevGrammar& g, const LexEntry* table, int vocab,
                        const int32_t* x, int B, int n, const int32_t* pos, int k, const int32_t* tok, int8_t* spec,
                        const WsPack& wsp);
void launch_select(dim3 grid, cudaStream_t st, const DevGrammar& g, const LexEntry* table, int vocab,
                   const int32_t* x, int B, int n, const int32_t* pos, int k, const int32_t* tok, const float* conf,
                   uint8_t* selected, const WsPack& wsp, const int8_t* spec, unsigned long long* stats);

// Alg. 1's sequential rejection fallback
void launch_fallback_init(int B, cudaStream_t st, int n, const int32_t* pos, int k, const float* conf, int K,
                          const int32_t* n_target, const uint8_t* selected, const uint8_t* valid, int32_t* filled,
                          uint8_t* rej, int32_t* fb, unsigned long long* active, unsigned long long* stats);
void launch_fallback_round(dim3 grid, cudaStream_t st, const DevGrammar& g, const LexEntry* table, int vocab,
                           const int32_t* x, int B, int n, const int32_t* pos, int k, const int32_t* cand,
                           const float* conf, int K, int m, const uint8_t* rej, const int32_t* fb, int32_t* res,
                           const WsPack& wsp, unsigned long long* stats);
void launch_fallback_resolve(int B, cudaStream_t st, int32_t* x, int n, const int32_t* pos, int k,
                             const int32_t* cand, int K, int m, uint8_t* rej, int32_t* fb, const int32_t* res,
                             int32_t* filled, unsigned long long* active, unsigned long long* stats);

// witness extraction (Sec. 4.4) from the forward charts of checks by region
void launch_witness(int B, cudaStream_t st, const DevGrammar& g, const SeqPack& sp, int32_t* terms, int cap,
                    int32_t* out_len, void* scratch, unsigned long long* stats);
size_t witness_scratch_bytes(int cap, int D, int W, int VW);  // scratch per sequence

// measurement builds (EPIC_PHASE_TIMERS): the walk's phase counters of one
// translation unit, added into out16 (reset: zeroed afterwards)
int phase_read_walk(unsigned long long* out16, int reset);
int phase_read_forward(unsigned long long* out16, int reset);
int phase_read_check_sm(unsigned long long* out16, int reset);
int phase_read_check_global(unsigned long long* out16, int reset);
int phase_read_good(unsigned long long* out16, int reset);

}  // namespace epic
