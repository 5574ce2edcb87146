/*
 * epic_measure.h -- measurement helper of the EPIC GB300 library.
 *
 * The paper has no counterpart: this is not part of the method.  It measures
 * the integer-pipe peak that the bit-parallel Earley sweeps are compared
 * against (their roofline denominator), on the current CUDA device.
 */
#ifndef EPIC_MEASURE_H_
#define EPIC_MEASURE_H_

#include "epic.h"

#ifdef __cplusplus
extern "C" {
#endif

/*
 * Peak rate of 32-bit word operations of the integer pipe: a full-occupancy
 * kernel of independent chains, each step one three-input logic operation
 * (LOP3) and one funnel shift (SHF), timed with CUDA events on cuda_stream
 * (best of three after a warm-up; synchronizes the stream).  One word
 * operation = one of those instructions on one 32-bit lane.  Writes the rate
 * (word operations per second) and the kernel's time in milliseconds (ms may
 * be NULL).  Returns 0, 1 for a NULL rate pointer, 4 if its 4-byte output
 * buffer cannot be allocated, 5 on a CUDA error.  Changes no clock or other
 * setting of the GPU.
 */
int epic_measure_int_peak(double* word_ops_per_s, double* ms, void* cuda_stream);

/*
 * Durations of the kernels that the last epic_validate_batch call on t
 * launched, in launch order (by region: the forward charts, the good masks,
 * the region checks; otherwise the one whole-graph walk kernel), followed by
 * the two kernels of the last epic_select_compatible_subset call on t (the
 * speculative first tests, then Alg. 4), each measured by CUDA events
 * recorded around its launch on the call's stream.  ms[i] receives kernel
 * i's milliseconds and names[i] (names may be NULL) a static kernel name.
 * Synchronizes on the last events.  Returns the number of kernels written
 * (at most cap), 0 before any call, -1 on a bad argument or a CUDA error.
 * The table owns the events; epic_validate_batch_noalloc records none.
 */
int epic_last_kernel_times(const epic_lexer_table* t, float* ms, const char** names, int cap);

#ifdef __cplusplus
}
#endif
#endif /* EPIC_MEASURE_H_ */
