/*
 * domino.h -- C ABI of libdomino.so: the per-decode-step hot path of DOMINO
 * ("Guiding LLMs The Right Way: Fast, Non-Invasive Constrained Generation")
 * on one GB300 GPU (sm_103a).
 *
 * The problem statement the calls follow (Alg. 1, Sec. 2): a checker C with
 * init / update / mask over a subword vocabulary V; C is a byte-level scanner
 * (Sec. 3.2) plus, for the context-free case, a bounded bracket-stack parser
 * (Sec. 3.4); the scanner x vocabulary table is precomputed offline
 * (Sec. 3.5), and the mask is applied to the logits before decoding
 * (Alg. 1, v' = m (.) v; decode = argmax).
 *
 * Conventions shared by every call
 *  - Return value: DOMINO_OK (0) or a negative DOMINO_E_* code.  Host-side
 *    argument checks are synchronous; nothing is launched when they fail.
 *  - "*_dev" pointers are device memory owned by the caller (e.g. torch
 *    tensors); kernels run asynchronously on `stream` (a cudaStream_t passed
 *    as void*, NULL = legacy default stream).  No call synchronises except the
 *    load calls, domino_get_device_error and domino_decode_step_host.
 *  - Mask layout: row b has W = ceil(V/32) uint32 words; token t is bit
 *    (t & 31) of word (t >> 5), least significant bit first; pad bits >= V
 *    are 0.
 *  - Stack word (uint64): bits 0..31 hold the bracket symbols with the top of
 *    the stack at bit 0 (a push shifts left and inserts at bit 0); bits 32..39
 *    hold the depth (0..max_depth); all other bits and the symbol bits at or
 *    above the depth are 0.  NULL stacks = every stack empty.
 *  - Invalid device inputs (state id outside [0, Q), a malformed stack word,
 *    a token id >= V in domino_advance) are treated as the dead configuration
 *    (all tokens rejected, next state 0) and set a bit of the sticky device
 *    error word read by domino_get_device_error.  No kernel traps.
 *  - A handle is not thread-safe; calls on one handle must be serialised by
 *    the caller, and their kernels must not overlap on the GPU either (issue
 *    them on one stream, or order the streams with events): the handle's
 *    scratch (the logits pass's partials and tickets, the fused decode's
 *    partials, the host-buffer step's staging) is shared by its calls.
 *    Different handles are independent.
 */
#ifndef DOMINO_H
#define DOMINO_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define DOMINO_OK 0
#define DOMINO_E_INVALID_ARG (-1)  /* bad pointer, size, id or automaton/vocabulary */
#define DOMINO_E_NOT_LOADED (-2)   /* vocabulary or automaton missing */
#define DOMINO_E_UNSUPPORTED (-3)  /* valid request this build does not implement */
#define DOMINO_E_OOM (-4)          /* device or host allocation failed */
#define DOMINO_E_CUDA (-5)         /* a CUDA runtime call failed */
#define DOMINO_E_NO_DEVICE (-6)    /* compute call on a host-only handle */

/* bits of the device error word */
#define DOMINO_DEVERR_BAD_STATE 1u
#define DOMINO_DEVERR_BAD_STACK 2u
#define DOMINO_DEVERR_BAD_TOKEN 4u
#define DOMINO_DEVERR_INTERNAL 8u   /* a kernel's own consistency check failed (a library bug) */

#define DOMINO_RULE_PUSH 1
#define DOMINO_RULE_POP 2
#define DOMINO_DTYPE_F32 0
#define DOMINO_DTYPE_BF16 1
#define DOMINO_MAX_DEPTH 32
#define DOMINO_MAX_STATES 65535

typedef struct domino_ctx* domino_t;

/* One bracket-stack rule (Sec. 3.4, the parser consulted on each terminal),
 * 20 bytes.  It fires on byte `byte` read in scanner state `state`, before
 * the scanner step:
 *   PUSH sym: rejected if depth == max_depth; else push sym and take the
 *             scanner transition delta[state][byte].
 *   POP sym:  rejected if depth == 0 or the top != sym; else pop, and the
 *             next state is next_if_empty / next_if_top0 / next_if_top1 by the
 *             symbol the pop reveals (delta[state][byte] is ignored). */
typedef struct {
    int32_t state;
    uint8_t byte;
    uint8_t kind; /* DOMINO_RULE_PUSH or DOMINO_RULE_POP */
    uint8_t sym;  /* 0 or 1 */
    uint8_t pad;  /* must be 0 */
    int32_t next_if_empty;
    int32_t next_if_top0;
    int32_t next_if_top1;
} domino_stack_rule;

/* What a handle holds (filled by domino_get_info). */
typedef struct {
    int32_t n_tokens;      /* V */
    int32_t n_words;       /* W = ceil(V/32) */
    int32_t eos_id;        /* -1: none */
    int32_t max_token_len; /* bytes */
    int32_t n_states;      /* Q */
    int32_t n_classes;     /* K, byte classes after compression */
    int32_t start_state;
    int32_t max_depth;
    int32_t n_rules;
    int32_t has_stack;     /* 1 when stack rules were loaded */
    int32_t table_in_smem; /* 1 when the transition table is staged in shared memory */
    int32_t device;        /* CUDA ordinal, -1 for a host-only handle */
    int64_t device_bytes;  /* device memory the handle owns */
    int32_t walk_tree;     /* 1: the mask step walks the vocabulary's prefix tree (domino_get_prefix_tree);
                              0: it walks every token on its own */
    int32_t tree_units;    /* subtrees the tree walk deals out (0 without a tree) */
} domino_info;

/* Creates a handle on CUDA device `cuda_device` (it becomes the current device
 * of the calling thread).  cuda_device = -1 creates a host-only handle that
 * validates and preprocesses loads but refuses every compute call with
 * DOMINO_E_NO_DEVICE.  *out is NULL on failure. */
int domino_create(domino_t* out, int32_t cuda_device);

/* Frees the handle and all device memory it owns (synchronises the device
 * first).  NULL is accepted. */
int domino_destroy(domino_t h);

/* Vocabulary V (Sec. 2, subword tokens; Fig. 3 c).  Token t is the byte
 * string bytes[offsets[t] .. offsets[t+1]) (host arrays, copied; offsets has
 * n_tokens + 1 entries, offsets[0] == 0, non-decreasing, each token <= 65535
 * bytes).  eos_id (-1: none) names the end-of-sequence token; its bytes are
 * ignored.  Replaces any earlier vocabulary; returns after the device copy is
 * complete.  1 <= n_tokens <= 2^24. */
int domino_load_vocab(domino_t h, const uint8_t* bytes, const int64_t* offsets, int32_t n_tokens,
                      int32_t eos_id);

/* Character scanner (Sec. 3.2, a DFA over bytes) and optional bracket rules
 * (Sec. 3.4).  delta is [n_states][256] int32 (host), live[q] != 0 marks states
 * from which acceptance is still reachable, accepting may be NULL (none).
 * Rejected (DOMINO_E_INVALID_ARG) unless: 1 <= n_states <= 65535; every id is
 * in [0, n_states); state 0 is non-live, absorbing and carries no rule; every
 * successor of a non-live state (including POP targets) is non-live;
 * accepting implies live; start_state is in range; rules name valid states,
 * kinds and symbols, pad == 0, at most one rule per (state, byte);
 * 0 <= max_depth <= 32.  Transitions into non-live states are redirected to
 * state 0 (exact early exit) and bytes that every state treats alike share a
 * byte class.  Returns after the device copy is complete. */
int domino_load_automaton(domino_t h, const int32_t* delta, int32_t n_states, const uint8_t* live,
                          const uint8_t* accepting, int32_t start_state, const domino_stack_rule* rules,
                          int32_t n_rules, int32_t max_depth);

int domino_get_info(domino_t h, domino_info* out);

/* Byte -> class id map of the loaded automaton (256 bytes, host). */
int domino_get_byte_classes(domino_t h, uint8_t* classes_out);

/* The prefix tree that the mask step walks (host copies, for inspection):
 * Alg. 2's subterminal tree (Sec. 3.3) over the byte-class strings of every
 * token except EOS and empty tokens.  Nodes are numbered in preorder, children
 * by class; node n is 8 uint32 words:
 *   [0] skip | cls << 24  (n's subtree is nodes [n, skip); cls: the class on
 *                          the edge into n, 0 for the root, node 0)
 *   [1] tok_lo  [2] n_end [3] tok_hi   (tokens_out[tok_lo, tok_lo + n_end) end
 *                          at n; tokens_out[tok_lo, tok_hi) are n's subtree's)
 *   [4] [5] the classes on the edges below n, a 64-bit set (when K <= 64)
 *   [6] [7] 0
 * tokens_out: original token ids in preorder.
 * upper_out [n_upper][2] = {node, depth}: the root and every node whose
 *   subtree has more than 64 nodes or more than 8 branching levels, in
 *   preorder; a row's configuration at each of them is computed first.
 * units_out [n_units][2] = {root node, index of its parent in upper_out}: the
 *   subtrees hanging off upper nodes, in preorder; each live (row, unit) pair
 *   is walked on its own.
 * sizes_out[4] (required) = {nodes, tokens, upper nodes, units}.  Each array
 * is copied up to its capacity (in entries) and may be NULL.  Available on
 * host-only handles too.  DOMINO_E_UNSUPPORTED: the tree exceeds 2^24 - 1
 * nodes (the mask step then walks every token on its own). */
int domino_get_prefix_tree(domino_t h, uint32_t* nodes_out, int64_t nodes_cap, int32_t* tokens_out,
                           int64_t tokens_cap, uint32_t* upper_out, int64_t upper_cap, uint32_t* units_out,
                           int64_t units_cap, int64_t* sizes_out);

/* Offline precompute (Alg. 2's "for every state q, for every token l,
 * traverse"; Sec. 3.5 "computed before inference starts"): for every state
 * q < Q, the mask row of q (mask_dev [Q][W]) and the next state of every token
 * (next_dev [Q][V] int32, 0 for rejected tokens; EOS keeps q).  Row q equals
 * domino_step_mask with states = {q} and empty stacks.  Either output may be
 * NULL, not both.  Pushdown automata: DOMINO_E_UNSUPPORTED (a row would
 * depend on the whole stack). */
int domino_precompute_table(domino_t h, int32_t* next_dev, uint32_t* mask_dev, void* stream);

/* C.mask() of Alg. 1 at lookahead k = infinity (Sec. 3.5; Definition
 * "minimally invasive", Sec. 2): for every sequence b < batch and token t,
 * t is allowed iff its bytes walked from (states_dev[b], stacks_dev[b])
 * through the scanner and bracket rules never reach a non-live state.  EOS is
 * allowed iff the state is accepting and the stack is empty (forced EOS,
 * Sec. 2; Fig. 3 e); other zero-length tokens are rejected.
 *   states_dev int32 [batch]; stacks_dev uint64 [batch] or NULL;
 *   mask_dev uint32 [batch][W] (written in full);
 *   next_dev int32 [batch][V] or NULL: end state of allowed tokens, 0 else.
 * batch = 0 is a no-op. */
int domino_step_mask(domino_t h, const int32_t* states_dev, const uint64_t* stacks_dev, int32_t batch,
                     uint32_t* mask_dev, int32_t* next_dev, void* stream);

/* Alg. 1 "v' = m (.) v; t = decode(v')" with greedy decode, fused: per row b,
 * over the allowed tokens only, m = max logit, argmax = the lowest token id
 * with logit m, lse = m + log(sum exp(logit - m)) (fp32 accumulation), and
 * logprob[t] = logit[t] - lse for allowed t, -inf for masked t.  A row with
 * no allowed token gives argmax -1, lse -inf and all log-probs -inf.
 *   logits_dev [batch] rows of V values (dtype DOMINO_DTYPE_F32 or
 *   DOMINO_DTYPE_BF16), row_stride_elems >= V apart; mask_dev [batch][W];
 *   argmax_dev int32 [batch] (required); lse_dev float [batch] or NULL;
 *   logprobs_dev float [batch][V] or NULL.
 * Logits must be finite.  Uses scratch memory owned by the handle. */
int domino_mask_logits(domino_t h, const void* logits_dev, int32_t dtype, int32_t batch,
                       int64_t row_stride_elems, const uint32_t* mask_dev, int32_t* argmax_dev, float* lse_dev,
                       float* logprobs_dev, void* stream);

/* C.update(o) of Alg. 1 for the token just decoded: walks tokens_dev[b] from
 * (states_dev[b], stacks_dev[b]).  tokens_dev[b] < 0 (no token) or == eos_id
 * ends the sequence and the next one starts from init: (start_state, empty).
 * A rejected token gives (0, empty).  Outputs may alias the inputs.
 * stacks_out may be NULL only when stacks_dev is NULL. */
int domino_advance(domino_t h, const int32_t* states_dev, const uint64_t* stacks_dev, const int32_t* tokens_dev,
                   int32_t batch, int32_t* states_out, uint64_t* stacks_out, void* stream);

/* One step of Alg. 1 on the device: C.mask(), the greedy decode and, when
 * states_out is given, C.update(o).  domino_step_mask's mask (written to
 * mask_dev as there), domino_mask_logits' argmax, lse and log-probs, with the
 * masked logits folded by the mask step itself, tile by tile, as soon as a
 * tile's bits are known (then a small per-row merge, which also advances each
 * row by its argmax as domino_advance does; the log-probs, when asked for,
 * take one more pass over the logits).
 *   states_dev, stacks_dev, batch: as domino_step_mask;
 *   logits_dev, dtype, row_stride_elems: as domino_mask_logits; may point to
 *   device memory or to pinned host memory;
 *   mask_dev uint32 [batch][W] (required); argmax_dev int32 [batch]
 *   (required); lse_dev float [batch] or NULL; logprobs_dev float [batch][V]
 *   or NULL (requires lse_dev);
 *   states_out int32 [batch] or NULL (no update), stacks_out uint64 [batch]
 *   (required with states_out when stacks_dev is given): the configurations
 *   after the decoded token; they may alias states_dev / stacks_dev.
 * The fused form needs bf16 rows on 16-byte boundaries; other inputs run the
 * two kernels one after the other.  Results equal domino_step_mask followed
 * by domino_mask_logits.  The first call with a larger batch allocates
 * scratch and synchronises `stream`; if `stream` is being captured into a
 * CUDA graph at that point, the call returns DOMINO_E_INVALID_ARG and
 * launches nothing (make one uncaptured call at the largest batch first). */
int domino_step_decode(domino_t h, const int32_t* states_dev, const uint64_t* stacks_dev, int32_t batch,
                       const void* logits_dev, int32_t dtype, int64_t row_stride_elems, uint32_t* mask_dev,
                       int32_t* argmax_dev, float* lse_dev, float* logprobs_dev, int32_t* states_out,
                       uint64_t* stacks_out, void* stream);

/* Alg. 1 with the greedy decode replaced by sampling: tokens_dev[b] is a draw
 * from softmax(logits / temperature) restricted to the allowed tokens of
 * mask_dev row b (-1 when nothing is allowed), by the Gumbel-max rule:
 * the argmax over allowed t of x_t * (1/T) + g_t, lowest index on ties, with
 * g_t = -ln(-ln(u_t)), u_t = (2k + 1) / 2^24, k = w >> 9, w = word (t mod 4)
 * of Philox4x32-10 (Salmon et al., SC'11) on the counter
 * (t / 4, b, offset low, offset high) under the key (seed low, seed high).
 * 1/T is one fp32 division and the score is formed with correctly rounded
 * fp32 operations (ln by the atanh series), so draws are reproducible bit for
 * bit by an independent implementation.  A caller passes a new offset per
 * decode step.  temperature must be finite and > 0.  Same logits and mask
 * layout as domino_mask_logits; uses the handle's scratch memory. */
int domino_mask_sample(domino_t h, const void* logits_dev, int32_t dtype, int32_t batch, int64_t row_stride_elems,
                       const uint32_t* mask_dev, float temperature, uint64_t seed, uint64_t offset,
                       int32_t* tokens_dev, void* stream);

/* Opportunistic masking (Sec. 3.5's speed-ups): the greedy token of a decode
 * step without computing every mask.  Per row: the unmasked argmax (lowest
 * index on ties) is proposed and checked with one walk from the row's
 * configuration; if allowed it is the masked argmax.  Only the rows whose
 * proposal is rejected get their full mask (domino_step_mask over the listed
 * rows) and the masked argmax.  tokens_dev[b] equals what
 * domino_step_mask + domino_mask_logits give (-1 when nothing is allowed).
 *   mask_scratch_dev uint32 [batch][W]: caller-owned scratch; its first
 *   n rows hold the masks of the fallback rows, in no fixed order.
 *   n_fallback_dev int32 [1] or NULL: receives the number of fallback rows.
 * No lse: the accepted rows' masks are never formed.  The first call with a
 * batch larger than any before allocates scratch and synchronises `stream`.
 * Invalid configurations behave as in domino_step_mask (error word, -1). */
int domino_opportunistic_step(domino_t h, const void* logits_dev, int32_t dtype, int32_t batch,
                              int64_t row_stride_elems, const int32_t* states_dev, const uint64_t* stacks_dev,
                              uint32_t* mask_scratch_dev, int32_t* tokens_dev, int32_t* n_fallback_dev,
                              void* stream);

/* Count-based speculative proposals (Sec. 3.6).  The count model
 * P(t | alpha, beta) = #chose(t) / #reached is keyed by the scanner state and
 * the top of the bracket stack: n_keys = Q for a DFA, 3 Q for a pushdown
 * automaton (key = state * 3 + top, top 0 for an empty stack, 1 + symbol
 * otherwise).  The caller owns the model, zero-initialised:
 *   counts_dev uint32 [n_keys][V]; best_dev uint64 [n_keys] (the most frequent
 *   token of each key, packed as count << 32 | (0xFFFFFFFF - token));
 *   reached_dev uint32 [n_keys].
 * domino_spec_update: token tokens_dev[b] >= 0 was chosen from configuration
 * b; rows with a negative token or an invalid configuration are skipped. */
int domino_spec_update(domino_t h, uint32_t* counts_dev, uint64_t* best_dev, uint32_t* reached_dev,
                       const int32_t* states_dev, const uint64_t* stacks_dev, const int32_t* tokens_dev,
                       int32_t batch, void* stream);

/* Up to s proposals per row: from the row's configuration, repeatedly the
 * key's most frequent token (lowest id on equal counts) while
 * count * 1000 >= min_permille * reached and reached > 0.  Each proposal is
 * walked and must be allowed from the current configuration; EOS (accepting
 * state, empty stack) is proposed and ends the chain.
 *   proposals_dev int32 [batch][s] (-1 past the chain); n_prop_dev [batch];
 *   chain_states_dev int32 [batch][s + 1], chain_stacks_dev uint64
 *   [batch][s + 1] or NULL: entry i is the configuration after i proposals
 *   (the last one repeated past the chain's end).  The verification is the
 *   ordinary mask step + decode over these batch * (s + 1) configurations
 *   (one LLM pass gives their logits). */
int domino_spec_propose(domino_t h, const uint64_t* best_dev, const uint32_t* reached_dev,
                        const int32_t* states_dev, const uint64_t* stacks_dev, int32_t batch, int32_t s,
                        int32_t min_permille, int32_t* proposals_dev, int32_t* n_prop_dev,
                        int32_t* chain_states_dev, uint64_t* chain_stacks_dev, void* stream);

/* Acceptance: decoded_dev int32 [batch][s + 1] is the constrained decode at
 * each chain configuration.  n_accept_dev[b] = the number of leading
 * proposals equal to it; tokens_out_dev[b] = the decode right after them and
 * states_out_dev / stacks_out_dev = the configuration it was decoded from
 * (apply it with domino_advance).  Any output except n_accept_dev may be
 * NULL. */
int domino_spec_accept(domino_t h, const int32_t* proposals_dev, const int32_t* n_prop_dev,
                       const int32_t* decoded_dev, const int32_t* chain_states_dev, const uint64_t* chain_stacks_dev,
                       int32_t batch, int32_t s, int32_t* n_accept_dev, int32_t* tokens_out_dev,
                       int32_t* states_out_dev, uint64_t* stacks_out_dev, void* stream);

/* Table-driven decode step, mask and decode (Sec. 3.5: the per-state masks
 * are computed before inference starts and looked up while decoding).  The
 * same fused masked argmax / lse / log-probs as domino_mask_logits, with row
 * b's mask taken from row states_dev[b] of table_mask_dev, the [Q][W] mask
 * table written by domino_precompute_table for this handle's automaton and
 * vocabulary.  A state outside [0, Q) reads as an empty row (argmax -1) and
 * sets DOMINO_DEVERR_BAD_STATE.  Pushdown automata: DOMINO_E_UNSUPPORTED
 * (their masks depend on the stack).  Uses the handle's scratch memory. */
int domino_mask_logits_table(domino_t h, const void* logits_dev, int32_t dtype, int32_t batch,
                             int64_t row_stride_elems, const uint32_t* table_mask_dev, const int32_t* states_dev,
                             int32_t* argmax_dev, float* lse_dev, float* logprobs_dev, void* stream);

/* Table-driven C.update() (Alg. 1): states_out[b] = table_next_dev[s][t] for
 * s = states_dev[b], t = tokens_dev[b], from the [Q][V] next-state table of
 * domino_precompute_table (0 for a rejected token).  t < 0 or t == eos_id:
 * the start state.  t >= V or s outside [0, Q): 0 and the device error word.
 * states_out may alias states_dev.  Pushdown automata: DOMINO_E_UNSUPPORTED. */
int domino_advance_table(domino_t h, const int32_t* table_next_dev, const int32_t* states_dev,
                         const int32_t* tokens_dev, int32_t batch, int32_t* states_out, void* stream);

/* One whole decode step from HOST memory (end-to-end use): logits (batch
 * rows of V values, dense) and the configurations come from host memory,
 * the mask step, the greedy decode and advance run on the device, and
 * tokens_host[b] (the argmax), lse_host (may be NULL) and the new
 * configurations are written back into states_host / stacks_host
 * (stacks_host may be NULL for a DFA); `stream` is synchronised before the
 * call returns.
 *   Logits are either copied in chunks of rows on a copy stream owned by the
 *   handle, overlapped with the mask step and each chunk's decode, or, when
 *   they are pinned (page-locked) bf16, possibly read in place by the mask
 *   step itself (domino_step_decode), so that only allowed logits cross the
 *   host link, during the walk.  For pinned bf16 logits the handle times both
 *   paths on its own calls and takes the faster, retiming the other every
 *   64th call; pageable or fp32 logits are always copied.
 * Device staging buffers are owned by the handle and grown on demand. */
int domino_decode_step_host(domino_t h, const void* logits_host, int32_t dtype, int32_t batch,
                            int32_t* states_host, uint64_t* stacks_host, int32_t* tokens_host, float* lse_host,
                            void* stream);

/* domino_mask_logits without a handle and without allocating anything.
 * Not a step of the paper (it has no counterpart there): it exists for callers
 * that cannot call cudaMalloc -- for example code running while another
 * component owns all of the device memory (a serving runtime whose caching
 * allocator has reserved the GPU), or code on a path where an allocation's
 * implicit device synchronisation is not acceptable -- and so cannot create a
 * handle either.
 *   Same arguments and results as domino_mask_logits, with the vocabulary size
 *   n_tokens passed directly; batch <= 512 (larger batches return
 *   DOMINO_E_INVALID_ARG: split them into calls of at most 512 rows).
 *   Scratch: a fixed 516 KiB array inside libdomino.so (per-row partials,
 *   tickets, temporary lse); every GPU that loads the library holds it until
 *   the process exits.  Nothing is allocated by this call: no cudaMalloc,
 *   cudaFree or allocating library routine.
 *   The first call on a device looks up the array's device address with that
 *   device current (the calling thread's current device); make that first
 *   call before any stream capture.
 *   All calls share the one array and each call clears the tickets it uses;
 *   calls that overlap on the GPU (other streams or host threads without
 *   ordering between them) race on it and corrupt each other's results, so
 *   order them, e.g. on one stream. */
int domino_mask_logits_noalloc(const void* logits_dev, int32_t dtype, int32_t batch, int32_t n_tokens,
                               int64_t row_stride_elems, const uint32_t* mask_dev, int32_t* argmax_dev,
                               float* lse_dev, float* logprobs_dev, void* stream);

/* Synchronises `stream`, returns the sticky device error word (DOMINO_DEVERR_*
 * bits, 0 = none) in *code and clears it. */
int domino_get_device_error(domino_t h, int32_t* code, void* stream);

/* Static text for a status code. */
const char* domino_status_string(int status);

#ifdef __cplusplus
}
#endif
#endif
