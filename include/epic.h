/*
 * epic.h -- C-ABI of the GB300 (sm_103a) hot path of EPIC
 * ("Efficient and Parallel Inference under CFG Constraints for Diffusion
 * Language Models", arXiv 2606.00722).
 *
 * One denoising step of a masked diffusion LM under a context-free grammar:
 * every (masked position, candidate token) pair is lexed through a memoized
 * token x lexer-state table and checked for completability by Earley-style
 * recognition over the partial output's lexeme graph; relaxed compatible
 * subset selection then picks a parallel commit that is re-checked jointly.
 *
 * Conventions (all calls):
 *   - Every d_* argument is a DEVICE pointer owned by the caller; every other
 *     pointer is host memory, read during the call only.
 *   - Token ids are 0..vocab-1; -1 in x means MASK.
 *   - Batch calls are asynchronous on `cuda_stream` (a cudaStream_t, NULL =
 *     legacy default stream).  Argument errors are detected on the host and
 *     returned synchronously before anything is enqueued.  Device-side
 *     capacity overflow is reported per check (value 2 in d_valid / d_selected)
 *     and counted in the statistics (epic_get_stats), never silently dropped.
 *   - The library owns the opaque objects and the device workspace they hold;
 *     a grammar or lexer table must not be destroyed while work that uses it
 *     is still in flight.  Calls that share one object must not overlap in
 *     time on different streams (they share its workspace).
 *   - There is no CPU fallback: when no CUDA device is usable the calls
 *     return EPIC_ERR_CUDA.
 */
#ifndef EPIC_H_
#define EPIC_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  EPIC_OK = 0,
  EPIC_ERR_INVALID_ARG = 1, /* bad pointer, size, id, position or NaN          */
  EPIC_ERR_GRAMMAR = 2,     /* malformed productions, or L(G) is empty          */
  EPIC_ERR_LEXER = 3,       /* malformed terminal regex, or it matches epsilon  */
  EPIC_ERR_OOM = 4,         /* host or device allocation failed                 */
  EPIC_ERR_CUDA = 5,        /* a CUDA call failed (no device, launch error ...) */
  EPIC_ERR_CAPACITY = 6,    /* a workload exceeded a device capacity limit      */
  EPIC_ERR_TIMEOUT = 7      /* a bounded device loop ran out of iterations      */
} epic_status;

typedef struct epic_grammar epic_grammar;         /* grammar + lexer DFA + device tables */
typedef struct epic_lexer_table epic_lexer_table; /* memoized token x state lex table    */

/*
 * Grammar description (host memory, copied by epic_grammar_create).
 * Symbols: terminals are 0..n_terminals-1, nonterminal j is n_terminals+j.
 * G = (V, Sigma_lex, P, S) of Sec. 3: the terminals are the lexemes.
 *
 * terminal_regex[t]: NUL-terminated byte regex.  Syntax: literal bytes;
 *   `\c` escapes any byte c (`\n`, `\t`, `\r` are newline, tab, CR);
 *   classes `[a-z_]`, negated `[^"]`, with ranges; `.` = any byte but '\n';
 *   grouping `( )`; alternation `|`; postfix `*`, `+`, `?`.
 * terminal_skip[t] = 1 drops the terminal from lexeme sequences (whitespace);
 *   a skipped terminal may not appear in a production.
 * Terminal priority is its index: when one lexeme matches several terminals
 * the lowest index wins.
 * Productions: lhs[p] in 0..n_nonterminals-1, right-hand side
 *   rhs[rhs_off[p] .. rhs_off[p+1]-1] (at most 62 symbols; empty = epsilon).
 */
typedef struct {
  int32_t n_terminals;
  const char* const* terminal_regex;
  const uint8_t* terminal_skip;
  int32_t n_nonterminals;
  int32_t start; /* nonterminal index of S */
  int32_t n_productions;
  const int32_t* lhs;
  const int32_t* rhs_off; /* [n_productions + 1] */
  const int32_t* rhs;
} epic_grammar_desc;

/*
 * Compile a grammar (Alg. 1, its set-up: compile the lexical map; the regular
 * cover of Sec. 4.3 / App. A.2 is derived from the same tables).  Builds the
 * union lexer DFA (minimized), trims unproductive and unreachable symbols,
 * numbers the dotted items and uploads the device tables to the current
 * CUDA device.  Errors: EPIC_ERR_INVALID_ARG (NULL / out-of-range ids),
 * EPIC_ERR_LEXER (bad regex, terminal matching epsilon), EPIC_ERR_GRAMMAR
 * (empty language), EPIC_ERR_CUDA / EPIC_ERR_OOM.  Synchronous.
 */
epic_status epic_grammar_create(const epic_grammar_desc* desc, epic_grammar** out);
void epic_grammar_destroy(epic_grammar* g);

/* Number of lexer DFA states (the states a span after a gap may
 * start in, Sec. 2 / Alg. 2), or -1 for NULL. */
int32_t epic_grammar_lexer_states(const epic_grammar* g);

/*
 * Build the memoized lexing table (Sec. 4.1, Alg. 2, App. D.1) on the device:
 * for every token t and lexer state q, the greedy transducer's run of
 * terminals over t's bytes and its end state (or DEAD).  The rule: at state q
 * reading byte c, follow delta(q, c) if defined; else, if q accepts, emit its
 * terminal and restart from delta(q0, c); else DEAD.  Skipped terminals are
 * not emitted.  Vocabulary (host): token t's bytes are
 * tok_bytes[tok_off[t] .. tok_off[t+1]-1]; every token has 1..64 bytes.
 * Table layout in HBM: [vocab][lexer states] entries of 16 bytes.  Enqueued
 * on cuda_stream; a token whose run exceeds 13 terminals is an
 * EPIC_ERR_CAPACITY error (checked when the call returns, which synchronizes
 * the stream once).
 */
epic_status epic_lexer_table_build(const epic_grammar* g, const int32_t* tok_off,
                                   const uint8_t* tok_bytes, int32_t vocab, void* cuda_stream,
                                   epic_lexer_table** out);
/*
 * The same lexing table built lazily (Alg. 2: lexing results are memoized as
 * they are first needed, not precomputed): no dense [vocab][states] table is
 * built; a device hash table of `capacity` entries (rounded up to a power of
 * two, at most 2^30) keyed by (token, lexer state) is filled by the walks,
 * each entry computed by the transducer above on its first lookup.  Every
 * call gives the same results as with the dense table.  A lookup that finds
 * no free slot within 64 probes, or finds its entry still being computed by
 * another thread after a bounded wait, computes the entry without storing it
 * (stats.lex_uncached).  Counters: stats.lex_lookups, stats.lex_misses (the
 * memo's hit rate is 1 - misses / lookups).  Errors as epic_lexer_table_build,
 * plus EPIC_ERR_CAPACITY when vocab x states does not fit 32-bit keys.
 * epic_lexer_table_copy is not available for lazy tables.  Synchronous.
 */
epic_status epic_lexer_table_build_lazy(const epic_grammar* g, const int32_t* tok_off,
                                        const uint8_t* tok_bytes, int32_t vocab, int64_t capacity,
                                        void* cuda_stream, epic_lexer_table** out);
void epic_lexer_table_destroy(epic_lexer_table* t);

/*
 * Copy lex-table entries of tokens [first_token, first_token + count) to host
 * memory (synchronous; an inspection aid of the table of Sec. 4.1, used by
 * the tests; dense tables only).  Entry (t, q) is 16 bytes:
 * uint16 end state (0xFFFF = DEAD), uint8 run length, uint8 terminals[13].
 * host_out must hold count * epic_grammar_lexer_states(g) * 16 bytes.
 */
epic_status epic_lexer_table_copy(const epic_lexer_table* t, int32_t first_token, int32_t count,
                                  void* host_out, size_t out_bytes);

/*
 * Batched validity checks (Sec. 3; Alg. 3 per check; Alg. 1's validity test):
 *   d_valid[b][j][c] = Valid_G(x_b, {(d_pos[b][j], d_cand[b][j][c])})
 *                    = 1[ L(G) cap C_{x_b (+) (pos, tok)} != empty ].
 * d_x [B][n] int32 (-1 = MASK); d_pos [B][k] int32, each a masked position of
 * its row; d_cand [B][k][K] int32 token ids; d_valid [B][k][K] uint8 output:
 * 0 invalid, 1 valid, 2 capacity overflow for that check (no result).
 * The partial-output graph: each maximal run of masks is one gap with a
 * Sigma_lex* self-loop (any terminal string, the mask count ignored); each
 * maximal run of tokens is a span lexed from q0 at the sequence start and
 * from every lexer state after a gap; before a gap a pending lexeme that some
 * byte could extend stays open (the gap absorbs it) and one that no byte can
 * extend is emitted; the last span is flushed at END.  Host-side errors:
 * EPIC_ERR_INVALID_ARG for sizes < 0 or NULL pointers with non-empty sizes.
 * Device-side: an unmasked position or an out-of-range token id yields 0 for
 * that check and counts in stats.bad_inputs.  Asynchronous.
 * Two strategies give identical results: one warp per check walking the
 * whole graph of x (+) (pos, tok); or, when item sets exceed 32 words or the
 * batch has more checks than resident walks, one forward chart of x per
 * sequence (with its graph and good-item masks) and one warp per check
 * walking only the candidate's region (stats.region_checks counts these).
 * The library's device workspaces grow on demand, each up to a share of the
 * GPU's memory (per-sequence charts 30 %, per-warp walks 25 %, block walks of
 * selection 25 %, never more than is free; EPIC_SEQ_WORKSPACE_MB,
 * EPIC_WARP_WORKSPACE_MB and EPIC_WORKSPACE_MB override, in MiB).  Smaller
 * budgets run fewer walks at a time; a failed allocation returns
 * EPIC_ERR_OOM.  A sequence whose chart does not fit walks its checks whole.
 */
epic_status epic_validate_batch(const epic_grammar* g, const epic_lexer_table* t,
                                const int32_t* d_x, int32_t B, int32_t n, const int32_t* d_pos,
                                int32_t k, const int32_t* d_cand, int32_t K, uint8_t* d_valid,
                                void* cuda_stream);

/*
 * epic_validate_batch without any device allocation.  The paper has no
 * counterpart: this entry point is for callers that cannot call cudaMalloc
 * -- a serving process that has handed all device memory to its own pool
 * (model weights, KV cache) before decoding starts, or a per-step decode
 * loop that must not take cudaMalloc's implicit device synchronization and
 * unbounded latency.  Same arguments and outputs as epic_validate_batch;
 * every check that neither call reports as overflow (2) gets the same bit.
 * It always walks each check's whole graph (never by region), so it may
 * additionally report 2 where epic_validate_batch answers, and it has two
 * extra capacity errors, both returned before anything is enqueued:
 *   - EPIC_ERR_CAPACITY when the grammar's item sets exceed 32 words and
 *     n > 128 (whole-graph walks of long rows of such grammars take
 *     seconds per check; use epic_validate_batch for them);
 *   - EPIC_ERR_CAPACITY when one walk's workspace, (8 n + 256) columns and
 *     256 n chart entries, does not fit in the array.
 * A check whose chart needs more than 256 n entries reports 2 (overflow).
 * Fewer walks run at once than in epic_validate_batch, so it is slower on
 * large batches.
 *
 * Scratch: a file-scope device array of 128 MiB inside the library, which
 * every GPU that loads the library holds until the process exits.
 * The first call on a device looks up the array's device address (once per
 * device, with that device current); make that first call before any
 * stream capture.  Every call on a device shares the one array and keeps
 * the last call's contents; the call clears what must start at zero.
 * Calls that overlap on the GPU (on different streams, or from different
 * threads) race on the array and must not be issued.
 */
epic_status epic_validate_batch_noalloc(const epic_grammar* g, const epic_lexer_table* t,
                                        const int32_t* d_x, int32_t B, int32_t n,
                                        const int32_t* d_pos, int32_t k, const int32_t* d_cand,
                                        int32_t K, uint8_t* d_valid, void* cuda_stream);

/*
 * Candidate set C of Alg. 1 (each position's best valid candidate), read as:
 * per proposed position, the highest-confidence candidate whose valid bit is
 * 1 (ties: lowest candidate index), else none.  d_cand [B][k][K] int32,
 * d_cand_conf [B][k][K] float32, d_valid [B][k][K] uint8; outputs d_tok [B][k]
 * int32 (-1 = none) and d_conf [B][k] float32.  Asynchronous.
 */
epic_status epic_pick_candidates(const int32_t* d_cand, const float* d_cand_conf,
                                 const uint8_t* d_valid, int32_t B, int32_t k, int32_t K,
                                 int32_t* d_tok, float* d_conf, void* cuda_stream);

/*
 * Relaxed compatible subset selection with exact shrink (Sec. 4.3, Alg. 4),
 * one sequence per CTA: C = the proposed (position, d_tok) pairs with
 * d_tok >= 0, sorted by descending d_conf (ties: ascending position);
 * B = ExactShrink(x, RelaxedSelect(x, C)) where RelaxedSelect's group test is
 * L(F_G) cap L(A_{x (+) C}) != empty on the flattened regular cover, and
 * ExactShrink's test is the exact check of the joint update.
 * d_selected [B][k] uint8: 1 = in the committed batch (|B| >= 2 or none),
 * 2 = capacity overflow for the sequence (nothing selected).  A NaN
 * confidence counts as bad input (nothing selected for that sequence).
 * Asynchronous.
 */
epic_status epic_select_compatible_subset(const epic_grammar* g, const epic_lexer_table* t,
                                          const int32_t* d_x, int32_t B, int32_t n,
                                          const int32_t* d_pos, int32_t k, const int32_t* d_tok,
                                          const float* d_conf, uint8_t* d_selected,
                                          void* cuda_stream);

/*
 * Commit (Alg. 1): d_x[b][d_pos[b][j]] = d_tok[b][j] where
 * d_selected[b][j] == 1.  Asynchronous.
 */
epic_status epic_commit(int32_t* d_x, int32_t B, int32_t n, const int32_t* d_pos, int32_t k,
                        const int32_t* d_tok, const uint8_t* d_selected, void* cuda_stream);

/*
 * Sequential rejection fallback (Alg. 1, the loop after the selected batch B
 * is committed, run when B fails its test or more commits are wanted): for each
 * of the max(0, d_n_target[b] - |B_b|) commits still wanted, take the
 * highest-confidence candidate over every proposed position and its K
 * candidates whose position is still masked in d_x and that was not
 * rejected; while x (+) c fails the exact test of Sec. 3, reject it (its
 * logit is suppressed) and take the next; commit the accepted one.  Ties in
 * confidence go to the lower position, then the lower candidate index; the
 * loop ends early when every candidate is rejected.
 * d_x [B][n] int32, updated in place (call after epic_commit of the selected
 * batch); d_pos [B][k], d_cand [B][k][K], d_cand_conf [B][k][K] float32 as
 * for epic_pick_candidates; d_n_target [B] int32 = n_t, the commits wanted
 * in this step; d_selected [B][k] (1 = in B) or NULL for |B| = 0;
 * d_valid [B][k][K] or NULL: epic_validate_batch's bits for the same
 * candidates on x before the selected batch was committed -- a candidate
 * whose bit is 0 is rejected without a test (it would fail it: a partial
 * output that is not completable stays so after more commits, App. D); the
 * result is the same with or without it.  Output d_filled [B][k] int32: the
 * token this call committed at slot j, else -1.  Each test is a whole-graph
 * walk of x (+) c by one CTA.  The loop runs in rounds: up to 16 CTAs per
 * sequence test its next candidates in order against the same x at once,
 * and the round is then read in that order (failures reject, the first pass
 * commits; after it, failures still reject and passes are tested again), so
 * the commits are the sequential loop's.
 * Errors: EPIC_ERR_INVALID_ARG (NULL pointers, sizes < 0),
 * EPIC_ERR_CAPACITY when k K > 4096.  A NaN confidence or a position out of
 * range leaves that sequence unchanged (stats.bad_inputs); a test that hits
 * a capacity limit rejects its candidate (stats.overflow).
 * Synchronizes with the stream once per round (it reads whether any
 * sequence still wants commits); stats.fallback_rounds counts the rounds.
 */
epic_status epic_fallback_commit(const epic_grammar* g, const epic_lexer_table* t, int32_t* d_x, int32_t B,
                                 int32_t n, const int32_t* d_pos, int32_t k, const int32_t* d_cand,
                                 const float* d_cand_conf, int32_t K, const int32_t* d_n_target,
                                 const uint8_t* d_selected, const uint8_t* d_valid, int32_t* d_filled,
                                 void* cuda_stream);

/*
 * Witness extraction for failure recovery (Sec. 4.4): for each row of d_x
 * [B][n], one completion -- a lexeme sequence of L(G) that the partial output
 * allows (C_x of Sec. 3) -- read off the row's forward Earley chart by a
 * top-down walk of the accepting item's derivation.  Output d_terms [B][cap]
 * int32: the terminal ids in order, each with bit 16 set when a mask run (a
 * gap) produces it (the recovery fills those runs), the rest being the
 * lexemes of the fixed text; d_len [B] int32: the length, -1 when the row is
 * not completable (no witness exists), -2 when its chart, the capacity cap or
 * the search bound was exceeded (stats.witness_failures counts searches that
 * found no derivation).  A nonterminal that a gap derives is written as one
 * of its shortest terminal strings.  Runs the forward charts of
 * epic_validate_batch's checks by region, then one warp per row.  Errors:
 * EPIC_ERR_INVALID_ARG (NULL pointers, sizes < 0, cap < 1).  Asynchronous.
 */
epic_status epic_extract_witness(const epic_grammar* g, const epic_lexer_table* t, const int32_t* d_x, int32_t B,
                                 int32_t n, int32_t* d_terms, int32_t cap, int32_t* d_len, void* cuda_stream);

/* Device counters accumulated since the object was created (or reset). */
typedef struct {
  uint64_t checks;           /* single-candidate validity checks run           */
  uint64_t valid;            /* of which valid                                 */
  uint64_t overflow;         /* checks or selections that hit a capacity limit */
  uint64_t bad_inputs;       /* unmasked positions / bad token ids / NaNs      */
  uint64_t columns;          /* Earley chart columns (graph nodes) processed   */
  uint64_t entries;          /* (node, origin) chart entries stored            */
  uint64_t cover_checks;     /* regular-cover group tests (Alg. 4, Relaxed)  */
  uint64_t exact_checks;     /* joint exact checks (Alg. 4, ExactShrink)     */
  uint64_t selected;         /* candidates committed by selection              */
  uint64_t region_checks;    /* of the checks, those answered by region walks
                                over a per-sequence forward chart            */
  uint64_t validate_kernels; /* kernel launches made by epic_validate_batch*  */
  uint64_t fallback_checks;  /* exact tests of the rejection fallback         */
  uint64_t fallback_commits; /* candidates it committed                       */
  uint64_t lex_lookups;      /* (token, lexer state) lookups of span lexing   */
  uint64_t lex_misses;       /* lazy tables: entries computed on first use    */
  uint64_t lex_uncached;     /* lazy tables: computed without being stored    */
  uint64_t witness_failures; /* witness searches that found no derivation     */
  uint64_t fallback_rounds;  /* rounds of epic_fallback_commit (2 launches each) */
} epic_stats;

/* Copy the counters (synchronizes the lexer table's last stream); out_bytes
 * must be >= sizeof(epic_stats).  reset != 0 zeroes them afterwards. */
epic_status epic_get_stats(const epic_lexer_table* t, epic_stats* out, size_t out_bytes, int reset);

const char* epic_status_string(epic_status s);

#ifdef __cplusplus
}
#endif
#endif /* EPIC_H_ */
