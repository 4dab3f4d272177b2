/*
 * grid.h -- C ABI of libgrid: GRID's cold full-vocabulary next-token mask on
 * NVIDIA GB300 (sm_103a).
 *
 * GRID ("Grammar-Railed Decoding", arXiv 2607.11951) masks an LLM's logits so
 * that every sampled token keeps the detokenized output a viable prefix of a
 * role- and schema-projected LALR(1) language.  This library implements the
 * paper's data-parallel hot path for a batch of B parser configurations:
 *
 *   grid_compile       grammar text + role projection + schema lexicons
 *                      -> LALR(1) ACTION/GOTO, union lexer DFA, identifier trie
 *                      (Sec. 2 "Three grammar layers"; Fig. 1 offline band)
 *   grid_load_vocab    token byte strings -> DFS-ordered byte trie with alias
 *                      classes (Def. 3)
 *   grid_specialize    upload + per-lexer-state context-independent (CI) token
 *                      classes (Sec. 4.2 CI/CD split), once per schema
 *   grid_configs_create / grid_advance
 *                      configurations kappa = (sigma, rho) (Def. 1) and the
 *                      batched per-token parser step (Sec. 6.1 step 7)
 *   grid_masks         M(kappa) for B configurations as a packed B x ceil(V/32)
 *                      uint32 bitmask (Def. 4, Sec. 4.1-4.2, Sec. 3.2 EOS gate)
 *   grid_apply_mask    logits <- -inf where the mask bit is 0 (Sec. 2,
 *                      "Masked decoding": masked_fill_(-inf))
 *
 * and around them, in the paper's decoding loop: grid_masks_apply (the mask
 * with the -inf fill in the same pass), grid_advance_masks (one decoding step:
 * the sampled tokens fed inside the mask step), grid_masks_static (the mask
 * with no device allocation), grid_cache_* / grid_masks_cached (the
 * configuration-keyed mask cache, Sec. 4.3), grid_forced_span (jump-forward,
 * Sec. 6.1 step 6), grid_reserve (the token-denominated termination reserve,
 * Sec. 5 Prop. 9) and grid_configs_enable_audit / grid_audit_* (the audit
 * chain, Sec. 6.4).
 *
 * Conventions
 *   - Every call returns 0 (GRID_OK) or a negative GRID_E_* code; the message of
 *     the last failure on the calling thread is available from grid_last_error.
 *   - Handles (grid_grammar, grid_vocab, grid_spec, grid_configs) are opaque and
 *     owned by the library; release them with the matching *_free call.
 *   - Pointers named d_* are CUDA device pointers owned by the caller.
 *     `stream` is a cudaStream_t passed as void*; NULL means the legacy default
 *     stream.  Calls that take a stream only enqueue work: they never
 *     synchronize and never allocate.  grid_specialize and
 *     grid_configs_create allocate device memory and synchronize.
 *   - Data-dependent failures are reported per row in a caller-supplied device
 *     int32 array d_status[B] with the GRID_ST_* codes below; they never trap
 *     and every device loop has a static bound.
 *   - Mask layout: bit t of row b is (d_mask[b*W + (t>>5)] >> (t&31)) & 1,
 *     W = ceil(V/32), LSB first.  Bits >= V, special tokens and (unless the EOS
 *     gate passes) EOS are 0.
 *
 * Grammar text format (one declaration per line, '#' comment lines):
 *   %token NAME "literal"   |  %token NAME /regex/    terminal; line order is the
 *                                                     priority of the contextual pick
 *   %ignore NAME /regex/                              ignored terminal (the set I)
 *   %category NAME                                    L3 lexicon category (<= 32)
 *   %start SYMBOL
 *   lhs -> X Y Z [@tag]                               production; %empty = epsilon
 * Regex syntax: literal bytes, escapes \n \t \r \xHH \<punct>, classes [...] with
 * ranges and leading ^, ( ), |, and postfix * + ?.  At most 127 terminals.
 *
 * Lexing semantics (readings of Sec. 2 and Sec. 4.1): maximal munch over the
 * regex union automaton; when a byte kills it, the pending lexeme r is emitted
 * and its candidates are the terminals accepting r (a category c also needs
 * r in W_c); the first candidate in priority order that is ignored or whose
 * simulated reduce chain reaches SHIFT is taken; otherwise the byte is rejected.
 * The killing byte is then fed from the start state.  The output is viable iff
 * the trailing lexeme is live for an ignored or allowed terminal (category
 * terminals also need r in Prefix(W_c)).
 */
#ifndef GRID_H
#define GRID_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- return codes ---- */
#define GRID_OK 0
#define GRID_E_INVALID_ARG (-1)          /* NULL handle, bad size, bad dtype            */
#define GRID_E_PARSE (-2)                /* grammar text or regex does not parse        */
#define GRID_E_LALR_CONFLICT (-3)        /* projected grammar is not LALR(1)            */
#define GRID_E_EMPTY_LANGUAGE (-4)       /* L(G_role) is empty (Sec. 2, L2 check)       */
#define GRID_E_LEXICON_NOT_IN_REGEX (-5) /* some w in W_c is not in R_c (Prop. 8 (d))   */
#define GRID_E_LEXER_PRECONDITION (-6)   /* lexer not accept-closed or not delimited    */
#define GRID_E_CUDA (-7)                 /* a CUDA runtime call failed                  */
#define GRID_E_TOO_LARGE (-8)            /* a table exceeds a documented limit          */
#define GRID_E_VOCAB (-9)                /* empty spelling, bad id, bad offsets         */

/* ---- per-row device status codes (d_status) ---- */
#define GRID_ST_OK 0
#define GRID_ST_NONVIABLE 1         /* the configuration is not a viable prefix      */
#define GRID_ST_STACK_OVERFLOW 2    /* a push would exceed max_depth                 */
#define GRID_ST_TOKEN_NOT_ALLOWED 3 /* grid_advance got a token outside the mask      */
#define GRID_ST_EMPTY_MASK 4        /* viable row, empty mask (a vocabulary that is   */
                                    /* not byte-complete; impossible with, Prop. 8)   */
#define GRID_ST_BOUND 5             /* a per-token overlay or reduce-chain bound hit  */
#define GRID_ST_COMPLETE 6          /* the row accepted EOS; its mask is all zero     */

/* ---- logits dtypes for grid_apply_mask ---- */
#define GRID_DTYPE_F32 0
#define GRID_DTYPE_BF16 1

typedef struct grid_grammar grid_grammar;
typedef struct grid_vocab grid_vocab;
typedef struct grid_spec grid_spec;
typedef struct grid_configs grid_configs;
typedef struct grid_cache grid_cache;

/* One L3 lexicon: the allowed words W_c of category terminal `category`
 * (Sec. 2, L3).  Word i is words[offsets[i] .. offsets[i+1]); host memory,
 * read during the call only. */
typedef struct grid_lexicon {
  const char* category;
  const uint8_t* words;
  const int64_t* offsets; /* n_words + 1 entries, non-decreasing, offsets[0] = 0 */
  int32_t n_words;
} grid_lexicon;

typedef struct grid_options {
  int32_t max_depth; /* stack capacity D per configuration (default 4096)          */
  int32_t reserved[7];
} grid_options;

/* Thread-local message of the last failure on this thread; copies at most n-1
 * bytes plus a NUL into buf and returns the full message length. */
size_t grid_last_error(char* buf, size_t n);

/* Sec. 2 (L1/L2/L3) and Fig. 1: parse `grammar_text`, keep the productions that
 * are untagged or whose tag is in the comma-separated `role_keep` list
 * (role_keep == NULL keeps every production), eliminate useless symbols, check
 * L(G_role) is non-empty, build the LALR(1) tables, the minimised union lexer
 * DFA and the identifier trie of the `n_lex` lexicons, and validate the
 * preconditions: W_c subset of R_c, an accept-closed lexer (no live
 * non-accepting state after an accepting one) and blank-delimited lexemes
 * (0x20 kills every accepting state of a non-ignored terminal, and some ignored
 * terminal accepts 0x20).  Host-only: touches no GPU.  `opt` may be NULL.
 * On success *out owns the grammar; free with grid_grammar_free. */
int grid_compile(const char* grammar_text, size_t len, const char* role_keep,
                 const grid_lexicon* lex, int32_t n_lex, const grid_options* opt,
                 grid_grammar** out);
void grid_grammar_free(grid_grammar* g);

/* Table sizes of a compiled grammar: out[0]=terminals incl. $end, out[1]=LALR
 * states, out[2]=nonterminals, out[3]=productions, out[4]=DFA states,
 * out[5]=byte classes, out[6]=lexicon-trie nodes, out[7]=categories. */
int grid_grammar_info(const grid_grammar* g, int64_t out[8]);

/* Debug/test view of the identifier trie over the union of the L3 lexicons
 * (host memory, n_nodes = out[6] of grid_grammar_info): nodes in BFS order
 * with each node's children in increasing byte order, node 0 the root (the
 * empty prefix); the children of node n are the edges cstart[n] ..
 * cstart[n+1]-1 (cstart: n_nodes + 1 entries), edge e spelling byte
 * cbyte[e] and leading to node cnode[e] (n_nodes - 1 edges); pcats[n] has
 * bit c set when node n's string is a prefix of a word of category c,
 * wcats[n] when it is a word of category c. */
int grid_grammar_lexicon_trie(const grid_grammar* g, int32_t* cstart, uint8_t* cbyte, int32_t* cnode,
                              uint32_t* pcats, uint32_t* wcats, int64_t n_nodes);

/* Def. 3: build the DFS-ordered byte trie of the vocabulary.  Token t has the
 * spelling bytes[offsets[t] .. offsets[t+1]) (host memory, read during the call).
 * `eos_id` and the `n_special` ids in `special_ids` are excluded from the trie
 * and permanently masked (EOS is set only by the EOS gate).  Distinct ids with
 * equal spellings form alias classes and always get equal bits.  An empty
 * spelling of a non-special id is GRID_E_VOCAB.  Host-only.  *out owns the
 * vocabulary; free with grid_vocab_free. */
int grid_load_vocab(const uint8_t* bytes, const int64_t* offsets, int32_t V, int32_t eos_id,
                    const int32_t* special_ids, int32_t n_special, grid_vocab** out);
void grid_vocab_free(grid_vocab* v);

/* Vocabulary facts: out[0]=V, out[1]=distinct spellings in the trie,
 * out[2]=1 if all 256 single-byte spellings are present (byte-complete,
 * Prop. 8 (a)), out[3]=total spelling bytes. */
int grid_vocab_info(const grid_vocab* v, int64_t out[4]);

/* Sec. 4.2 + Sec. 8 (cold-schema specialization): upload grammar and
 * vocabulary tables to the current CUDA device and precompute, for every state
 * of the lexer DFA, the context-independent class of every spelling (the
 * spellings whose verdict is a function of the allowed-terminal set alone).
 * The grammar and vocabulary must outlive the spec.  Allocates device memory,
 * runs kernels on `stream` and synchronizes it.  *out owns the device tables;
 * free with grid_spec_free. */
int grid_specialize(const grid_grammar* g, const grid_vocab* v, void* stream, grid_spec** out);
void grid_spec_free(grid_spec* s);

/* Facts about a spec (synchronous): out[0]=precomputed lexer states (CI
 * tables), out[1]=CI class ids, out[2]=spellings of the start state walked
 * byte by byte at mask time (more stack-dependent events than one record
 * holds), out[3]=such entries over all tables, out[4]=bytes of the tables
 * staged in shared memory (0 = not staged), out[5]=verdict classes (distinct
 * event records of stack-dependent spellings) over all tables, out[6]=flags:
 * bit 0 = CI classes enabled (off when the 16-bit class codes cannot hold
 * every class id: 2 x DFA states x 2^categories >= 65531), bit 1 = a verdict
 * class's index rides in its id's class code (off when class ids, 5 special
 * codes and the largest table's verdict classes exceed 65535; then a per-id
 * index table is read), out[7]=distinct spellings. */
int grid_spec_info(const grid_spec* s, int64_t out[8]);

/* Create B configurations, all at the start configuration (empty output),
 * with the device scratch that grid_masks needs for B rows (1 <= B <= 65535;
 * GRID_E_TOO_LARGE above).  Allocates device memory and synchronizes.  Free
 * with grid_configs_free. */
int grid_configs_create(const grid_spec* s, int32_t B, grid_configs** out);
void grid_configs_free(grid_configs* c);

/* Reset every row of `c` to the start configuration (enqueued on `stream`). */
int grid_configs_reset(const grid_spec* s, grid_configs* c, void* stream);

/* Sec. 6.1 step 7: per row b, feed the tokens d_tokens[b*n_steps + k],
 * k = 0..n_steps-1, in order (a negative id is a no-op).  Each token must be in
 * the row's current mask: its bytes go through the lexer (maximal munch,
 * parser-viable pick) and the emitted terminals are shifted/reduced on the
 * row's stack; EOS (when the gate passes) completes the row.  `in` and `out`
 * may be the same object (in place) or two configurations of the same B
 * (out-of-place: `in` is not modified).  On a token outside the mask the row
 * keeps its configuration as of the last accepted token and d_status[b] =
 * GRID_ST_TOKEN_NOT_ALLOWED (also for out-of-range ids and special tokens);
 * a full stack gives GRID_ST_STACK_OVERFLOW; a completed row gives
 * GRID_ST_COMPLETE.  Enqueue only. */
int grid_advance(const grid_spec* s, const grid_configs* in, grid_configs* out,
                 const int32_t* d_tokens, int32_t n_steps, int32_t* d_status, void* stream);

/* Def. 4: write M(kappa_b) for every row of `c` into d_mask[B][W] (device,
 * W = ceil(V/32), 4-byte aligned).  A viable row whose mask would be empty gets
 * GRID_ST_EMPTY_MASK; a completed row gets an all-zero mask and
 * GRID_ST_COMPLETE.  Uses the scratch held by `c`, so calls on the same
 * configurations object must not overlap on the GPU.  Enqueue only. */
int grid_masks(const grid_spec* s, const grid_configs* c, uint32_t* d_mask, int32_t* d_status,
               void* stream);

/* grid_masks and grid_apply_mask in one pass: writes M(kappa_b) into d_mask
 * exactly as grid_masks does and, in the same kernel that packs each mask
 * word, sets d_logits[b*row_stride + t] to -inf where bit t is 0 (accepted
 * values bit-identical), as grid_apply_mask would on the finished mask; the
 * logits of a completed row become all -inf.  Fusing the fill into the
 * packing saves re-reading the mask and one launch per decoding step (Sec. 2
 * masked decoding, Def. 4).  d_logits: device memory of `dtype`
 * (GRID_DTYPE_F32 or GRID_DTYPE_BF16), row_stride >= V elements.  The same
 * scratch and overlap rule as grid_masks.  Enqueue only. */
int grid_masks_apply(const grid_spec* s, const grid_configs* c, uint32_t* d_mask, int32_t* d_status,
                     void* d_logits, int32_t dtype, int64_t row_stride, void* stream);

/* One decoding step in one launch sequence (Sec. 6.1 steps 7 then 1-5):
 * grid_advance of d_tokens (n_steps per row) from `in` into `out`, then
 * grid_masks of `out` -- or grid_masks_apply when d_logits is not NULL
 * (dtype and row_stride as there; d_logits NULL: no fill, dtype and
 * row_stride unused); with `cache` (a cache of `s`, or NULL) through the
 * mask cache as grid_masks_cached.  The advance runs inside the mask step's first kernel,
 * one row per block, so that a row's mask preparation starts as soon as its
 * own token is fed.  The configurations and masks are those of grid_advance
 * followed by grid_masks(_apply); d_status[b] is the advance's status when
 * row b's token was refused (GRID_ST_TOKEN_NOT_ALLOWED, GRID_ST_STACK_OVERFLOW,
 * GRID_ST_BOUND, GRID_ST_COMPLETE: the row keeps its configuration as of the
 * last accepted token and is masked there), else the mask step's.  `in` and
 * `out` follow grid_advance's rules (same B and D, audit on both or neither;
 * in == out advances in place); the scratch and overlap rule of grid_masks
 * apply to `out`.  Enqueue only. */
int grid_advance_masks(const grid_spec* s, const grid_configs* in, grid_configs* out, grid_cache* cache,
                       const int32_t* d_tokens, int32_t n_steps, uint32_t* d_mask, int32_t* d_status,
                       void* d_logits, int32_t dtype, int64_t row_stride, void* stream);

/* Measurement hook: with n_events == 5, every later grid_masks on `c` records
 * events[0..4] (cudaEvent_t, created by the caller) on its stream before its
 * first kernel and after each of its four kernels (per-row allowed sets, EOS
 * gate, allowed sets after one shift and class selections; filtering of
 * what the walk evaluates; walk and verdict classes; id-order packing), so
 * that cudaEventElapsedTime between neighbours gives each kernel's duration.
 * n_events == 0 stops the recording.  The caller keeps the events alive while
 * they are set. */
int grid_configs_set_events(grid_configs* c, void* const* events, int32_t n_events);

/* ---- configuration-keyed mask cache (Sec. 4.3, Def. T1 key, Prop. OBL-KEY1) ----
 * A cache holds, per key, the context-independent part of a mask: the bits
 * of the token ids whose verdict the CI classes decide, and which ids are
 * the stack-dependent residue.  The key is (kind, lexer state, whether the
 * pending lexeme's forced emission succeeds, A(sigma), A(sigma')): kind 1
 * marks identifier positions (a lexer state where a lexicon category is
 * live), a distinct key type, whose continuing ids are always residue, so a
 * generic entry is never consulted at an identifier position; the spec (its
 * grammar, role and schema) scopes the whole cache.  The residue (verdict
 * classes and byte walks) and the EOS gate are never cached and are computed
 * on every step, so a hit changes no bit of any mask (OBL-KEY1; the tests
 * compare cache-on with cache-off over randomized replays).  Entries are
 * filled by the step that first meets a key (an empty slot is claimed; the
 * slot is the key's hash modulo n_entries, no eviction) and read from the
 * next step on; the content is a function of the key, so concurrent fills of
 * one key write identical words. */

/* Allocate a cache of n_entries (a power of two, <= 2^20) entries of
 * 64 + 8 * ceil(V/32) bytes for spec `s` (which must outlive it).
 * Synchronizes.  Free with grid_cache_free. */
int grid_cache_create(const grid_spec* s, int32_t n_entries, grid_cache** out);
void grid_cache_free(grid_cache* c);

/* Empty every entry and zero the counters (enqueued on `stream`). */
int grid_cache_clear(grid_cache* c, void* stream);

/* Counters (synchronous): out[0] lookups, out[1] hits, out[2] entries
 * claimed for filling, out[3] entries ready. */
int grid_cache_stats(const grid_cache* c, int64_t out[4]);

/* grid_masks (d_logits == NULL) or grid_masks_apply (d_logits of `dtype`,
 * row_stride >= V) reading and filling `cache`: the same masks, statuses and
 * logits bit for bit, with the context-independent part of each row taken
 * from the cache on a hit.  Calls that use one cache must not overlap on the
 * GPU.  Enqueue only. */
int grid_masks_cached(const grid_spec* s, const grid_configs* c, grid_cache* cache, uint32_t* d_mask,
                      int32_t* d_status, void* d_logits, int32_t dtype, int64_t row_stride, void* stream);

/* Measurement hook: with d_counters (device memory, 6 x u64, zeroed by the
 * caller) set, every later mask step on `s` adds to it the work of its walk
 * kernel in the units of the walk's algorithmic cost: [0] lexer steps (trie
 * node visits of byte walks), [1] ACTION lookups (reduce-chain steps, for one
 * terminal or a set of terminals at once), [2] GOTO lookups, [3] verdict-class
 * events evaluated; and what it evaluated: [4] verdict-class records (one per
 * row, context and surviving class: the verdict classes of Sec. 4.2 decided by
 * the step), [5] spellings walked byte by byte.  Counting slows that kernel
 * down; time steps without it.  NULL stops the counting. */
int grid_spec_set_work_counters(grid_spec* s, unsigned long long* d_counters);

/* grid_masks without any allocation.  The paper has no counterpart: this is
 * an interface for callers that cannot allocate device memory when they need
 * a mask, e.g. a serving engine whose memory pool has reserved the device up
 * front, or that cannot pay for the device-wide synchronization of freeing
 * memory in the middle of a decoding step.  Such a caller keeps the B parser
 * configurations in device memory it owns and passes them as arrays with the
 * layout grid_configs_export reports for one row:
 *   d_stack     uint16 LALR(1) states, row b at d_stack[b*stack_stride ...],
 *               bottom first, d_depth[b] entries used;
 *               stack_stride must equal the grammar's max_depth
 *   d_depth, d_dfa_state, d_lex_node, d_flags   int32[B] (flags bit 0 =
 *               complete)
 * Each row must hold a configuration this library produced (read back with
 * grid_configs_export, or copied from such a row); other contents are not
 * checked.  Outputs and status codes are those of grid_masks.
 *
 * The step's scratch is one fixed 8 MiB array in the library's device image,
 * reserved on every device that loads the library until the process exits;
 * a (spec, B) whose scratch does not fit is rejected with GRID_E_TOO_LARGE
 * before anything is enqueued (the scratch grows with B and with the spec:
 * two V-bit verdict bitmaps and the verdict-class survivor lists per row,
 * about 175 KB per row for the SQL grammar at V = 151,936, so about 48 rows).
 * The first call on a device looks up the array's device address (set-up,
 * once per device, with that device current); make that first call before any
 * stream capture.  The address is kept for the life of the process, so the
 * device's primary context must stay alive between calls (no
 * cudaDeviceReset), and calls must run with that primary context current.
 * B <= 65535 (GRID_E_TOO_LARGE above, as for any scratch that does not fit).  Every call on a device shares the array: calls whose kernels
 * overlap on the GPU (other streams, other threads) race and corrupt each
 * other's masks, so serialize them.  Each call clears what must start at zero
 * itself.  The spec must live on the current device.  Enqueue only. */
int grid_masks_static(const grid_spec* s, const uint16_t* d_stack, const int32_t* d_depth,
                      const int32_t* d_dfa_state, const int32_t* d_lex_node, const int32_t* d_flags, int32_t B,
                      int32_t stack_stride, uint32_t* d_mask, int32_t* d_status, void* stream);

/* Sec. 6.1 step 6, jump-forward: per row, while the mask of the row's
 * configuration admits exactly one token id (EOS included), that token is
 * forced: it is appended to the row's span and the row is advanced by it (in
 * place), up to max_span tokens (0 <= max_span <= 4096).  On return d_span
 * [B][max_span] holds each row's forced ids in order (-1 after its span),
 * d_span_len[B] their count, and d_mask / d_status the mask and status of the
 * row's final configuration, as grid_masks writes them; a forced token that
 * cannot be advanced stops the row with grid_advance's status.  Runs one mask
 * step per span position (max_span + 1 in all) whatever the spans' lengths,
 * so choose max_span by the longest forced run worth taking.  With audit
 * enabled on `c`, every forced token is audited (record kind 1, see
 * grid_audit_append) into d_records [B][max_span] records of 80 bytes (row
 * b's k-th forced token at d_records + (b * max_span + k) * 80); d_records
 * must then be given, and must be NULL otherwise.  Uses the scratch held by
 * `c`; enqueue only. */
int grid_forced_span(const grid_spec* s, grid_configs* c, int32_t max_span, uint32_t* d_mask, int32_t* d_span,
                     int32_t* d_span_len, int32_t* d_status, uint8_t* d_records, void* stream);

/* Sec. 5 Prop. 9 (Termination) and Sec. 6.1 step 3: the token-denominated
 * reserve of every row -- the cheapest legal completion of the row's output
 * plus EOS, counted in vocabulary tokens -- so that a decoding loop whose
 * remaining budget falls to the reserve plus a safety margin writes that
 * completion instead of sampling (every stop then lies in L).
 * Cost model (the paper's: terminal costs in tokens, summed over a
 * completion): terminal tau is written as a blank and its lexeme l(tau) (the
 * shortest, then bytewise smallest, string whose first emission candidate is
 * tau; a lexicon word for a category), split greedily into vocabulary tokens;
 * the pending lexeme either ends as it stands or is first extended, in
 * single-byte tokens, to one live terminal's shortest lexeme, then ends by
 * the blank of the first rendering (or the lexer state's separator byte, a
 * token of its own); the completion's terminals minimise the summed
 * rendering lengths exactly (over the LR items of the stack, see
 * grid_span.cu).  Writes d_cost[b] = tokens of the completion including EOS
 * (0 for a completed row, -1 when none exists) and the tokens themselves to
 * d_tokens[b*cap ...] (-1 after them); d_status[b] = GRID_ST_OK,
 * GRID_ST_COMPLETE, GRID_ST_NONVIABLE (no completion under this cost model)
 * or GRID_ST_BOUND (the completion is longer than cap -- d_cost still holds
 * its length -- or the search space of a very deep stack ran out).  With
 * d_budget given, d_fire[b] = 1 when d_budget[b] <= d_cost[b] + safety (the
 * reserve trigger), else 0.  Uses the scratch held by `c`; enqueue only. */
int grid_reserve(const grid_spec* s, const grid_configs* c, int32_t* d_cost, int32_t* d_tokens, int32_t cap,
                 int32_t* d_status, const int32_t* d_budget, int32_t safety, int32_t* d_fire, void* stream);

/* ---- audit chain (Sec. 6.4) ----
 * Every decoding step of a row appends a record, chained by BLAKE2b-128 from
 * a genesis constant.  Record layout (80 bytes, little-endian):
 *   0  u64 step           records of the row so far (0, 1, 2, ...)
 *   8  u64 config_hash    rolling hash of the top stack node of the
 *                         configuration the step's mask was computed at:
 *                         H(root) = 0, H(node) = low 64 bits (LE) of
 *                         BLAKE2b-128(u64 H(parent) || u32 kind || u32 id),
 *                         (kind, id) the symbol entering the node: (0,
 *                         terminal index) or (1, rank of the nonterminal's
 *                         name in byte order among the grammar's nonterminals)
 *   16 u8[16] mask id     BLAKE2b-128("GRIDmask" || u32 V || u32 chunks ||
 *                         BLAKE2b-128 of each 1,024-byte chunk of the mask row)
 *   32 i32 token          the sampled or forced id (the seal: stop reason)
 *   36 u32 blocked        ids < V the mask rejects (the seal: mode flags)
 *   40 u32 kind           caller's label (0 sampled, 1 forced, 2 EOS tail by
 *                         convention), 3 = seal
 *   44 u8[16] prev        the previous record's hash (genesis for step 0)
 *   60 u32 zero
 *   64 u8[16] hash        BLAKE2b-128 of bytes 0..59
 * The hashes are kept on the device next to the configurations; appending
 * costs O(1) per push and O(V/32) per record, independent of the position. */

/* Enable auditing on `c`: allocates the node hashes (B x max_depth x 8 bytes)
 * and the per-row chain heads, hashes every row's current stack and starts a
 * fresh chain per row.  Synchronizes.  Afterwards grid_advance on `c` keeps
 * the node hashes (both configurations of an advance must have audit on, or
 * neither), and grid_configs_reset restarts every row's chain. */
int grid_configs_enable_audit(const grid_spec* s, grid_configs* c, void* stream);

/* Append one record per row b with d_tokens[b] >= 0 (other rows are left
 * alone) to d_records + b * 80: the configuration hash of the row as it is
 * now, the id of d_mask's row b (which must be the mask of that
 * configuration), the token, the rejected-id count and `kind` (>= 0).  Call
 * it after the mask step and before grid_advance with the same token.
 * Enqueue only. */
int grid_audit_append(const grid_spec* s, grid_configs* c, const uint32_t* d_mask, const int32_t* d_tokens,
                      int32_t kind, uint8_t* d_records, void* stream);

/* Seal every row's log: a record of kind 3 with the final configuration's
 * hash, the spec's fingerprint in place of the mask id, d_reason[b] (the stop
 * reason, caller-defined) as the token and mode_flags as the blocked count,
 * written to d_records + b * 80.  Enqueue only. */
int grid_audit_seal(const grid_spec* s, grid_configs* c, const int32_t* d_reason, uint32_t mode_flags,
                    uint8_t* d_records, void* stream);

/* Chain head (16 bytes) and record count of one row (synchronous). */
int grid_audit_head(const grid_configs* c, int32_t row, uint8_t* head, uint64_t* n_records);

/* Host-side check of one row's log of n records (host memory, in order): each
 * record's step is its index, its prev is the previous record's hash (or
 * `genesis`, NULL = the library's constant), and its hash matches its bytes.
 * Returns the index of the first record that fails, or -1 when all pass
 * (a negative GRID_E_* on bad arguments). */
int64_t grid_audit_verify(const uint8_t* records, int64_t n, const uint8_t* genesis);

/* The genesis constant: BLAKE2b-128 of the 24 bytes "GRID audit chain genesis". */
int grid_audit_genesis(uint8_t* out16);

/* BLAKE2b (RFC 7693, unkeyed) of n bytes of host memory, out_bytes in 1..64;
 * the hash the audit chain is built from. */
int grid_blake2b(const void* data, size_t n, uint8_t* out, int32_t out_bytes);

/* Fingerprint (16 bytes) of exactly one of: a grammar (BLAKE2b-128 of
 * "GRIDgram", u64 text length, the text, the role list as passed (u64 length
 * and bytes, or u64 all ones when NULL), u64 lexicon count, per lexicon in
 * call order u64 name length, name, u64 word count, u64 length and bytes of
 * each word, then u64 max_depth), a vocabulary (BLAKE2b-128 of "GRIDvoca", u64
 * V, i64 eos, u64 special count, i64 each special id, then u64 length and
 * bytes of every token), or a spec (BLAKE2b-128 of "GRIDspec" and the two).
 * The other two pointers must be NULL. */
int grid_fingerprint(const grid_grammar* g, const grid_vocab* v, const grid_spec* s, uint8_t* out16);

/* Sec. 2 masked decoding: for b < B, t < V, set d_logits[b*row_stride + t] to
 * -inf (fp32 0xFF800000 / bf16 0xFF80) where mask bit t of row b is 0; accepted
 * values are left bit-identical.  d_logits is device memory of `dtype`
 * (GRID_DTYPE_F32 or GRID_DTYPE_BF16); row_stride >= V elements; B <= 65535
 * (GRID_E_TOO_LARGE above).  In place, enqueue only. */
int grid_apply_mask(const uint32_t* d_mask, void* d_logits, int32_t dtype, int32_t B, int32_t V,
                    int64_t row_stride, void* stream);

/* Debug/test view of row `row` (synchronous device-to-host copy): the stack
 * (up to `cap` entries, bottom first), its depth, the lexer DFA state and
 * lexicon-trie node of the pending lexeme, and flags (bit 0 = complete). */
int grid_configs_export(const grid_configs* c, int32_t row, int32_t* stack, int32_t cap,
                        int32_t* depth, int32_t* dfa_state, int32_t* lex_node, int32_t* flags);

#ifdef __cplusplus
}
#endif

#endif /* GRID_H */
