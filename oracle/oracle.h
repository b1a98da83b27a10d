/*
 * oracle.h -- plain CPU oracle for DOMINO's per-step constrained-decoding path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may link, load or
 * call this code: it is used by the tests, by the smoke check and by the
 * benchmark's CPU-baseline leg.  It shares no code, header, table or constant
 * with the CUDA library; the two are compared against each other.
 *
 * What it computes (the paper's definitions, written out; no blocking, no
 * byte-class compression, no dead-state canonicalisation):
 *
 *   token check  (Sec. 3.5, k = infinity; Definition "minimally invasive",
 *                 Sec. 2): a token t is allowed from configuration (s, stack)
 *                 iff walking its bytes through the scanner and bracket parser
 *                 never leaves the live (co-reachable) states; the walk's end
 *                 state is the token's next state.  EOS is allowed iff s is
 *                 accepting and the stack is empty (Sec. 2, forced EOS;
 *                 Fig. 3 (e)).  Every other zero-length token is rejected.
 *   pushdown     (Sec. 3.4, parser consulted on every terminal): a stack rule
 *                 (state, byte) PUSH g / POP g fires before the byte's scanner
 *                 step; POP checks the top and picks the next state from the
 *                 symbol the pop reveals.
 *   mask_logits  (Alg. 1, v' = m (.) v, then decode): masked maximum, lowest
 *                 index on ties, log-sum-exp and log-probabilities in double.
 *   advance      (Alg. 1, C.update(o)): the chosen token's walk; EOS or "no
 *                 token" ends the sequence and the next one starts from init.
 *   spec_*       (Sec. 3.6, count-based speculative proposals): counts of
 *                 the tokens chosen in each (scanner state, parser sub-state);
 *                 up to s tokens proposed by following the most frequent
 *                 choice while its share is large enough; proposals accepted
 *                 up to the first position where the constrained decode
 *                 disagrees.
 *   mask_sample  (Alg. 1, decode by sampling instead of the argmax): the
 *                 Gumbel-max rule over the allowed tokens, with uniforms from
 *                 the Philox4x32-10 counter-based generator (Salmon et al.,
 *                 SC'11).  The score that decides the sample is formed in fp32
 *                 with one fixed sequence of correctly rounded operations.
 *
 * All arrays are host memory owned by the caller.
 */
#ifndef DOMINO_ORACLE_H
#define DOMINO_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { ORACLE_PUSH = 1, ORACLE_POP = 2 };
enum { ORACLE_F32 = 0, ORACLE_BF16 = 1 };

/* One bracket rule, 20 bytes, little-endian. */
typedef struct {
    int32_t state;
    uint8_t byte;
    uint8_t kind;          /* ORACLE_PUSH or ORACLE_POP */
    uint8_t sym;           /* 0 or 1 */
    uint8_t pad;
    int32_t next_if_empty; /* POP: next state when the pop empties the stack */
    int32_t next_if_top0;  /* POP: next state when symbol 0 is revealed */
    int32_t next_if_top1;  /* POP: next state when symbol 1 is revealed */
} oracle_rule;

typedef struct oracle_problem oracle_problem;

/* Copies everything it is given.  delta is [n_states][256] int32, live and
 * accepting are [n_states] (accepting may be NULL: none).  Returns NULL on a
 * malformed problem (ids out of range, two rules on one (state, byte),
 * max_depth outside 0..32). */
oracle_problem* oracle_new(const uint8_t* bytes, const int64_t* offsets, int32_t n_tokens, int32_t eos_id,
                           const int32_t* delta, int32_t n_states, const uint8_t* live,
                           const uint8_t* accepting, const oracle_rule* rules, int32_t n_rules,
                           int32_t max_depth);
void oracle_free(oracle_problem* p);

/* One (configuration, token) check.  stack is the packed boundary word
 * (bits 0..31 symbols with the top at bit 0, bits 32..39 depth).
 * Returns 1 allowed (outputs written), 0 rejected, -1 invalid configuration. */
int oracle_check_token(const oracle_problem* p, int32_t state, uint64_t stack, int32_t token,
                       int32_t* next_state, uint64_t* next_stack);

/* mask: [batch][ceil(V/32)] bit t%32 of word t/32, pad bits 0.  next: [batch][V]
 * (NULL: not written), 0 for rejected tokens.  stacks may be NULL (all empty).
 * Returns the number of rows whose configuration was invalid (all rejected). */
int64_t oracle_step_mask(const oracle_problem* p, const int32_t* states, const uint64_t* stacks,
                         int32_t batch, uint32_t* mask, int32_t* next, int32_t n_threads);

/* Work of the plain definition: the number of (byte, transition) steps that
 * checking every token from every row takes, each walk counted up to and
 * including the byte that rejects it (EOS and empty tokens take none).
 * Invalid rows count 0.  Used to state the algorithmic work of a mask step. */
int64_t oracle_walk_steps(const oracle_problem* p, const int32_t* states, const uint64_t* stacks,
                          int32_t batch, int32_t n_threads);

/* Per row of logits ([batch] rows of n_tokens values, row_stride elements
 * apart; dtype ORACLE_F32 or ORACLE_BF16 raw bits): argmax [batch] (-1 when
 * every token is masked), lse [batch] (NULL: skipped), logprobs
 * [batch][n_tokens] (NULL: skipped; -inf for masked tokens). */
void oracle_mask_logits(const void* logits, int32_t dtype, int32_t batch, int32_t n_tokens,
                        int64_t row_stride, const uint32_t* mask, int32_t* argmax, double* lse,
                        double* logprobs, int32_t n_threads);

/* Philox4x32-10: ten rounds on the 128-bit counter ctr under the 64-bit key
 * (key0, key1); the four output words replace ctr. */
void oracle_philox4x32_10(uint32_t ctr[4], uint32_t key0, uint32_t key1);

/* Natural logarithm of a positive normal float: x = 2^e m with m in
 * [sqrt(1/2), sqrt(2)), ln x = e ln 2 + 2 atanh((m - 1) / (m + 1)), atanh by
 * its odd power series to the z^11 term, every step a correctly rounded fp32
 * operation. */
float oracle_ln_f32(float x);

/* Sampling decode (Alg. 1 with the greedy argmax replaced by a draw from the
 * masked softmax at temperature T): tokens[b] = argmax over allowed t of
 * x_t * (1/T) + g_t, lowest index on ties, -1 when nothing is allowed.
 * g_t = -ln(-ln(u_t)) (a Gumbel variate, so the argmax is distributed as
 * softmax(x / T) over the allowed tokens); u_t = (2k + 1) / 2^24 with
 * k = w >> 9 and w word (t mod 4) of Philox4x32-10 on the counter
 * (t / 4, b, offset low, offset high) under the key (seed low, seed high).
 * All arithmetic of the score is fp32.  temperature > 0. */
void oracle_mask_sample(const void* logits, int32_t dtype, int32_t batch, int32_t n_tokens, int64_t row_stride,
                        const uint32_t* mask, float temperature, uint64_t seed, uint64_t offset, int32_t* tokens,
                        int32_t n_threads);

/* Count-based speculation (Sec. 3.6).  The count model is keyed by
 * (alpha, beta) = (scanner state, top of the bracket stack): key = state for a
 * plain DFA, state * 3 + top for a pushdown automaton, top = 0 for an empty
 * stack, 1 + symbol otherwise. */
typedef struct oracle_spec oracle_spec;
oracle_spec* oracle_spec_new(const oracle_problem* p);
void oracle_spec_free(oracle_spec* sp);

/* After a decode step: the token tokens[b] (>= 0) was chosen from
 * configuration b: #reached(key) += 1 and #chose(key, token) += 1.  Rows with
 * a negative token or an invalid configuration are skipped. */
void oracle_spec_update(oracle_spec* sp, const int32_t* states, const uint64_t* stacks, const int32_t* tokens,
                        int32_t batch);

/* Up to s proposals per row: from the row's configuration, repeatedly take
 * the key's most frequent token (lowest id on equal counts) while
 * count * 1000 >= min_permille * #reached(key) and #reached > 0; a proposed
 * token must be allowed from the current configuration (the walk is taken and
 * the configuration advanced); EOS is proposed and ends the chain.
 *   proposals [batch][s] (-1 past n_prop[b]); n_prop [batch];
 *   chain_states / chain_stacks [batch][s + 1]: entry i is the configuration
 *   after the first i proposals (entries past n_prop[b] repeat the last one);
 *   chain_stacks may be NULL. */
void oracle_spec_propose(const oracle_spec* sp, const int32_t* states, const uint64_t* stacks, int32_t batch,
                         int32_t s, int32_t min_permille, int32_t* proposals, int32_t* n_prop,
                         int32_t* chain_states, uint64_t* chain_stacks);

/* Verification: decoded [batch][s + 1] holds the constrained decode at each
 * chain configuration; n_accept[b] = the number of leading proposals equal to
 * it (at most n_prop[b]). */
void oracle_spec_accept(const int32_t* proposals, const int32_t* n_prop, const int32_t* decoded, int32_t batch,
                        int32_t s, int32_t* n_accept);

/* Alg. 1 update: states_out/stacks_out may alias the inputs.  tokens[b] < 0 or
 * == eos_id: (start_state, empty).  A rejected token: (0, empty).  A token id
 * >= V or an invalid configuration: (0, empty), counted in the return value. */
int64_t oracle_advance(const oracle_problem* p, const int32_t* states, const uint64_t* stacks,
                       const int32_t* tokens, int32_t batch, int32_t start_state, int32_t* states_out,
                       uint64_t* stacks_out);

#ifdef __cplusplus
}
#endif
#endif
