/*
 * oracle.c -- plain CPU oracle (TEST INFRASTRUCTURE ONLY; see oracle.h).
 *
 * Written for a reader checking it against the paper: tokens are kept as
 * their byte strings, the scanner as the raw [Q][256] table, the bracket
 * stack as an array of symbols.  Loops are the definitions, nothing more.
 * OpenMP (when compiled in) only splits independent rows across threads.
 */
#include "oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_MAX_DEPTH 32

struct oracle_problem {
    int32_t n_tokens, eos_id, n_states, max_depth, n_rules;
    uint8_t* bytes;      /* all token bytes */
    int64_t* offsets;    /* [n_tokens + 1] */
    int32_t* delta;      /* [n_states][256] */
    uint8_t* live;       /* [n_states] */
    uint8_t* accepting;  /* [n_states] */
    oracle_rule* rules;  /* [n_rules] */
    int32_t* rule_at;    /* [n_states][256]: index into rules or -1 */
};

static void* dup_bytes(const void* src, size_t n) {
    void* d = malloc(n ? n : 1);
    if (d && n) memcpy(d, src, n);
    return d;
}

oracle_problem* oracle_new(const uint8_t* bytes, const int64_t* offsets, int32_t n_tokens, int32_t eos_id,
                           const int32_t* delta, int32_t n_states, const uint8_t* live,
                           const uint8_t* accepting, const oracle_rule* rules, int32_t n_rules,
                           int32_t max_depth) {
    if (n_tokens < 0 || n_states < 1 || max_depth < 0 || max_depth > ORACLE_MAX_DEPTH) return NULL;
    if (eos_id >= n_tokens) return NULL;
    for (int64_t i = 0; i < (int64_t)n_states * 256; i++)
        if (delta[i] < 0 || delta[i] >= n_states) return NULL;
    oracle_problem* p = (oracle_problem*)calloc(1, sizeof(*p));
    p->n_tokens = n_tokens;
    p->eos_id = eos_id;
    p->n_states = n_states;
    p->max_depth = max_depth;
    p->n_rules = n_rules > 0 ? n_rules : 0;
    p->offsets = (int64_t*)dup_bytes(offsets, sizeof(int64_t) * (size_t)(n_tokens + 1));
    p->bytes = (uint8_t*)dup_bytes(bytes, (size_t)offsets[n_tokens]);
    p->delta = (int32_t*)dup_bytes(delta, sizeof(int32_t) * (size_t)n_states * 256);
    p->live = (uint8_t*)dup_bytes(live, (size_t)n_states);
    p->accepting = (uint8_t*)calloc((size_t)n_states, 1);
    if (accepting) memcpy(p->accepting, accepting, (size_t)n_states);
    p->rules = (oracle_rule*)dup_bytes(rules, sizeof(oracle_rule) * (size_t)(n_rules > 0 ? n_rules : 0));
    p->rule_at = (int32_t*)malloc(sizeof(int32_t) * (size_t)n_states * 256);
    for (int64_t i = 0; i < (int64_t)n_states * 256; i++) p->rule_at[i] = -1;
    for (int32_t r = 0; r < n_rules; r++) {
        const oracle_rule* R = &rules[r];
        int bad = R->state < 0 || R->state >= n_states || (R->kind != ORACLE_PUSH && R->kind != ORACLE_POP) ||
                  R->sym > 1;
        if (!bad && R->kind == ORACLE_POP)
            bad = R->next_if_empty < 0 || R->next_if_empty >= n_states || R->next_if_top0 < 0 ||
                  R->next_if_top0 >= n_states || R->next_if_top1 < 0 || R->next_if_top1 >= n_states;
        int32_t* slot = bad ? NULL : &p->rule_at[(int64_t)R->state * 256 + R->byte];
        if (bad || *slot != -1) {   /* malformed, or two rules on one (state, byte) */
            oracle_free(p);
            return NULL;
        }
        *slot = r;
    }
    return p;
}

void oracle_free(oracle_problem* p) {
    if (!p) return;
    free(p->bytes); free(p->offsets); free(p->delta); free(p->live); free(p->accepting);
    free(p->rules); free(p->rule_at);
    free(p);
}

/* The bracket stack as the parser sees it: sym[0] is the bottom. */
typedef struct {
    int depth;
    uint8_t sym[ORACLE_MAX_DEPTH];
} stack_t_;

/* Boundary word -> stack.  Returns 0 when the word is not a valid stack. */
static int decode_stack(uint64_t w, int max_depth, stack_t_* st) {
    uint64_t depth = (w >> 32) & 0xFF;
    uint64_t bits = w & 0xFFFFFFFFull;
    if ((w >> 40) != 0 || depth > (uint64_t)max_depth) return 0;
    if (depth < 32 && (bits >> depth) != 0) return 0;   /* symbols above the depth must be zero */
    st->depth = (int)depth;
    for (int i = 0; i < st->depth; i++)                  /* top symbol at bit 0 */
        st->sym[i] = (uint8_t)((bits >> (st->depth - 1 - i)) & 1);
    return 1;
}

static uint64_t encode_stack(const stack_t_* st) {
    uint64_t bits = 0;
    for (int i = 0; i < st->depth; i++) bits = (bits << 1) | st->sym[i];
    return ((uint64_t)st->depth << 32) | bits;
}

static int config_valid(const oracle_problem* p, int32_t state, uint64_t stack, stack_t_* st) {
    if (state < 0 || state >= p->n_states) return 0;
    return decode_stack(stack, p->max_depth, st);
}

/* Walk one token from (s, st); st is updated in place.  Returns 1 when the
 * token is allowed (Sec. 3.5 at k = infinity), with *end the state reached.
 * *steps (when not NULL) counts the bytes taken, the last one included. */
static int walk_token(const oracle_problem* p, int32_t s, stack_t_* st, int32_t t, int32_t* end,
                      int64_t* steps) {
    int64_t lo = p->offsets[t], hi = p->offsets[t + 1];
    if (t == p->eos_id) {                         /* forced EOS: accepting and nothing left open */
        *end = s;
        return p->accepting[s] && st->depth == 0;
    }
    if (hi == lo) return 0;                       /* other empty tokens never advance the output */
    for (int64_t i = lo; i < hi; i++) {
        uint8_t c = p->bytes[i];
        if (steps) (*steps)++;
        int32_t r = p->rule_at[(int64_t)s * 256 + c];
        if (r < 0) {
            s = p->delta[(int64_t)s * 256 + c];
        } else if (p->rules[r].kind == ORACLE_PUSH) {
            if (st->depth == p->max_depth) return 0;          /* bounded stack is full */
            st->sym[st->depth++] = p->rules[r].sym;
            s = p->delta[(int64_t)s * 256 + c];
        } else {                                              /* POP */
            if (st->depth == 0 || st->sym[st->depth - 1] != p->rules[r].sym) return 0;
            st->depth--;
            if (st->depth == 0) s = p->rules[r].next_if_empty;
            else if (st->sym[st->depth - 1] == 0) s = p->rules[r].next_if_top0;
            else s = p->rules[r].next_if_top1;
        }
        if (!p->live[s]) return 0;                /* no continuation can reach acceptance */
    }
    *end = s;
    return 1;
}

int oracle_check_token(const oracle_problem* p, int32_t state, uint64_t stack, int32_t token,
                       int32_t* next_state, uint64_t* next_stack) {
    stack_t_ st;
    if (!config_valid(p, state, stack, &st) || token < 0 || token >= p->n_tokens) return -1;
    int32_t end = 0;
    if (!walk_token(p, state, &st, token, &end, NULL)) return 0;
    if (next_state) *next_state = end;
    if (next_stack) *next_stack = encode_stack(&st);
    return 1;
}

int64_t oracle_step_mask(const oracle_problem* p, const int32_t* states, const uint64_t* stacks,
                         int32_t batch, uint32_t* mask, int32_t* next, int32_t n_threads) {
    const int32_t V = p->n_tokens;
    const int64_t W = ((int64_t)V + 31) / 32;
    int64_t invalid = 0;
#ifdef _OPENMP
    if (n_threads < 1) n_threads = 1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(n_threads) reduction(+ : invalid)
#endif
    for (int32_t b = 0; b < batch; b++) {
        uint32_t* mrow = mask + (int64_t)b * W;
        int32_t* nrow = next ? next + (int64_t)b * V : NULL;
        memset(mrow, 0, sizeof(uint32_t) * (size_t)W);
        if (nrow) memset(nrow, 0, sizeof(int32_t) * (size_t)V);
        stack_t_ st0;
        if (!config_valid(p, states[b], stacks ? stacks[b] : 0, &st0)) {
            invalid++;
            continue;
        }
        for (int32_t t = 0; t < V; t++) {
            stack_t_ st = st0;
            int32_t end = 0;
            if (walk_token(p, states[b], &st, t, &end, NULL)) {
                mrow[t / 32] |= 1u << (t % 32);
                if (nrow) nrow[t] = end;
            }
        }
    }
    return invalid;
}

int64_t oracle_walk_steps(const oracle_problem* p, const int32_t* states, const uint64_t* stacks,
                          int32_t batch, int32_t n_threads) {
    int64_t total = 0;
#ifdef _OPENMP
    if (n_threads < 1) n_threads = 1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(n_threads) reduction(+ : total)
#endif
    for (int32_t b = 0; b < batch; b++) {
        stack_t_ st0;
        if (!config_valid(p, states[b], stacks ? stacks[b] : 0, &st0)) continue;
        int64_t n = 0;
        for (int32_t t = 0; t < p->n_tokens; t++) {
            stack_t_ st = st0;
            int32_t end = 0;
            walk_token(p, states[b], &st, t, &end, &n);
        }
        total += n;
    }
    return total;
}

static double logit_value(const void* logits, int32_t dtype, int64_t i) {
    if (dtype == ORACLE_BF16) {
        uint32_t u = (uint32_t)((const uint16_t*)logits)[i] << 16;   /* bf16 -> f32 is exact */
        float f;
        memcpy(&f, &u, sizeof f);
        return (double)f;
    }
    return (double)((const float*)logits)[i];
}

void oracle_mask_logits(const void* logits, int32_t dtype, int32_t batch, int32_t n_tokens,
                        int64_t row_stride, const uint32_t* mask, int32_t* argmax, double* lse,
                        double* logprobs, int32_t n_threads) {
    const int64_t W = ((int64_t)n_tokens + 31) / 32;
#ifdef _OPENMP
    if (n_threads < 1) n_threads = 1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(n_threads)
#endif
    for (int32_t b = 0; b < batch; b++) {
        const uint32_t* mrow = mask + (int64_t)b * W;
        const int64_t base = (int64_t)b * row_stride;
        /* v' = m (.) v with -inf on masked tokens; decode = argmax (lowest index on ties) */
        double m = -INFINITY;
        int32_t best = -1;
        for (int32_t t = 0; t < n_tokens; t++) {
            if (!((mrow[t / 32] >> (t % 32)) & 1)) continue;
            double x = logit_value(logits, dtype, base + t);
            if (x > m) { m = x; best = t; }
        }
        argmax[b] = best;
        double l = -INFINITY;
        if (best >= 0) {
            double sum = 0.0;
            for (int32_t t = 0; t < n_tokens; t++)
                if ((mrow[t / 32] >> (t % 32)) & 1) sum += exp(logit_value(logits, dtype, base + t) - m);
            l = m + log(sum);
        }
        if (lse) lse[b] = l;
        if (logprobs) {
            double* lp = logprobs + (int64_t)b * n_tokens;
            for (int32_t t = 0; t < n_tokens; t++)
                lp[t] = ((mrow[t / 32] >> (t % 32)) & 1) ? logit_value(logits, dtype, base + t) - l : -INFINITY;
        }
    }
}

/* ---- sampling (Gumbel-max over the masked logits) ------------------------ */

void oracle_philox4x32_10(uint32_t ctr[4], uint32_t key0, uint32_t key1) {
    for (int round = 0; round < 10; round++) {
        if (round > 0) {                          /* key schedule: add the Weyl constants */
            key0 += 0x9E3779B9u;
            key1 += 0xBB67AE85u;
        }
        uint64_t p0 = (uint64_t)0xD2511F53u * ctr[0];
        uint64_t p1 = (uint64_t)0xCD9E8D57u * ctr[2];
        uint32_t y0 = (uint32_t)(p1 >> 32) ^ ctr[1] ^ key0;
        uint32_t y1 = (uint32_t)p1;
        uint32_t y2 = (uint32_t)(p0 >> 32) ^ ctr[3] ^ key1;
        uint32_t y3 = (uint32_t)p0;
        ctr[0] = y0;
        ctr[1] = y1;
        ctr[2] = y2;
        ctr[3] = y3;
    }
}

float oracle_ln_f32(float x) {
    uint32_t bits;
    memcpy(&bits, &x, sizeof bits);
    int32_t e = (int32_t)((bits >> 23) & 0xFFu) - 127;
    uint32_t mb = (bits & 0x7FFFFFu) | 0x3F800000u;   /* mantissa in [1, 2) */
    float m;
    memcpy(&m, &mb, sizeof m);
    if (m > 0x1.6a09e6p+0f) {                        /* move m into [sqrt(1/2), sqrt(2)) */
        m = m * 0.5f;
        e = e + 1;
    }
    float num = m - 1.0f;
    float den = m + 1.0f;
    float z = num / den;
    float z2 = z * z;
    float poly = 0x1.745d18p-4f;                    /* 1/11 */
    poly = fmaf(poly, z2, 0x1.c71c72p-4f);           /* 1/9 */
    poly = fmaf(poly, z2, 0x1.24924ap-3f);           /* 1/7 */
    poly = fmaf(poly, z2, 0x1.99999ap-3f);           /* 1/5 */
    poly = fmaf(poly, z2, 0x1.555556p-2f);           /* 1/3 */
    poly = fmaf(poly, z2, 1.0f);
    float two_z = z + z;
    float r = two_z * poly;                          /* 2 atanh(z) = ln m */
    float ef = (float)e;
    float lo = fmaf(ef, -0x1.05c61p-29f, r);         /* e ln2 in two parts */
    return fmaf(ef, 0x1.62e43p-1f, lo);
}

void oracle_mask_sample(const void* logits, int32_t dtype, int32_t batch, int32_t n_tokens, int64_t row_stride,
                        const uint32_t* mask, float temperature, uint64_t seed, uint64_t offset, int32_t* tokens,
                        int32_t n_threads) {
    const int64_t W = ((int64_t)n_tokens + 31) / 32;
    const float inv_t = 1.0f / temperature;
    const uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
#ifdef _OPENMP
    if (n_threads < 1) n_threads = 1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(n_threads)
#endif
    for (int32_t b = 0; b < batch; b++) {
        const uint32_t* mrow = mask + (int64_t)b * W;
        const int64_t base = (int64_t)b * row_stride;
        float best_score = -INFINITY;
        int32_t best = -1;
        for (int32_t t = 0; t < n_tokens; t++) {
            if (!((mrow[t / 32] >> (t % 32)) & 1)) continue;
            uint32_t c[4] = {(uint32_t)t / 4u, (uint32_t)b, (uint32_t)offset, (uint32_t)(offset >> 32)};
            oracle_philox4x32_10(c, k0, k1);
            uint32_t k = c[t % 4] >> 9;
            float u = (float)(2u * k + 1u) * 0x1p-24f;       /* exact: an odd integer below 2^24 */
            float e1 = -oracle_ln_f32(u);                    /* Exp(1) variate */
            float g = -oracle_ln_f32(e1);                    /* Gumbel variate */
            float x = (float)logit_value(logits, dtype, base + t);
            float scaled = x * inv_t;
            float score = scaled + g;
            if (score > best_score) {
                best_score = score;
                best = t;
            }
        }
        tokens[b] = best;
    }
}

/* ---- count-based speculation (Sec. 3.6) --------------------------------- */

struct oracle_spec {
    const oracle_problem* p;
    int32_t n_keys;
    int64_t* reached;     /* [n_keys] */
    int32_t* len;         /* [n_keys]: distinct tokens seen */
    int32_t* cap;
    int32_t** tok;        /* [n_keys][len] token ids */
    int64_t** cnt;        /* [n_keys][len] times chosen */
};

static int spec_key(const oracle_problem* p, int32_t state, const stack_t_* st) {
    if (p->n_rules == 0) return state;
    int top = st->depth == 0 ? 0 : 1 + st->sym[st->depth - 1];
    return state * 3 + top;
}

oracle_spec* oracle_spec_new(const oracle_problem* p) {
    oracle_spec* sp = (oracle_spec*)calloc(1, sizeof *sp);
    if (!sp) return NULL;
    sp->p = p;
    sp->n_keys = p->n_rules == 0 ? p->n_states : p->n_states * 3;
    sp->reached = (int64_t*)calloc((size_t)sp->n_keys, sizeof(int64_t));
    sp->len = (int32_t*)calloc((size_t)sp->n_keys, sizeof(int32_t));
    sp->cap = (int32_t*)calloc((size_t)sp->n_keys, sizeof(int32_t));
    sp->tok = (int32_t**)calloc((size_t)sp->n_keys, sizeof(int32_t*));
    sp->cnt = (int64_t**)calloc((size_t)sp->n_keys, sizeof(int64_t*));
    return sp;
}

void oracle_spec_free(oracle_spec* sp) {
    if (!sp) return;
    for (int32_t k = 0; k < sp->n_keys; k++) {
        free(sp->tok[k]);
        free(sp->cnt[k]);
    }
    free(sp->reached);
    free(sp->len);
    free(sp->cap);
    free(sp->tok);
    free(sp->cnt);
    free(sp);
}

void oracle_spec_update(oracle_spec* sp, const int32_t* states, const uint64_t* stacks, const int32_t* tokens,
                        int32_t batch) {
    const oracle_problem* p = sp->p;
    for (int32_t b = 0; b < batch; b++) {
        int32_t t = tokens[b];
        stack_t_ st;
        if (t < 0 || t >= p->n_tokens || !config_valid(p, states[b], stacks ? stacks[b] : 0, &st)) continue;
        int key = spec_key(p, states[b], &st);
        sp->reached[key]++;
        int32_t i = 0;
        while (i < sp->len[key] && sp->tok[key][i] != t) i++;
        if (i == sp->len[key]) {                      /* first time t is chosen here */
            if (sp->len[key] == sp->cap[key]) {
                int32_t nc = sp->cap[key] ? 2 * sp->cap[key] : 4;
                sp->tok[key] = (int32_t*)realloc(sp->tok[key], sizeof(int32_t) * (size_t)nc);
                sp->cnt[key] = (int64_t*)realloc(sp->cnt[key], sizeof(int64_t) * (size_t)nc);
                sp->cap[key] = nc;
            }
            sp->tok[key][i] = t;
            sp->cnt[key][i] = 0;
            sp->len[key]++;
        }
        sp->cnt[key][i]++;
    }
}

void oracle_spec_propose(const oracle_spec* sp, const int32_t* states, const uint64_t* stacks, int32_t batch,
                         int32_t s, int32_t min_permille, int32_t* proposals, int32_t* n_prop,
                         int32_t* chain_states, uint64_t* chain_stacks) {
    const oracle_problem* p = sp->p;
    for (int32_t b = 0; b < batch; b++) {
        int32_t state = states[b];
        uint64_t word = stacks ? stacks[b] : 0;
        int32_t n = 0;
        stack_t_ st;
        int ok = config_valid(p, state, word, &st);
        while (ok && n < s) {
            int key = spec_key(p, state, &st);
            int64_t reached = sp->reached[key];
            if (reached == 0) break;
            int32_t best = -1;
            int64_t best_c = 0;
            for (int32_t i = 0; i < sp->len[key]; i++) {   /* most frequent, lowest id on ties */
                if (sp->cnt[key][i] > best_c || (sp->cnt[key][i] == best_c && sp->tok[key][i] < best)) {
                    best_c = sp->cnt[key][i];
                    best = sp->tok[key][i];
                }
            }
            if (best < 0 || best_c * 1000 < (int64_t)min_permille * reached) break;
            if (best == p->eos_id) {                       /* EOS is proposed and ends the chain */
                if (!(p->accepting[state] && st.depth == 0)) break;
                proposals[(int64_t)b * s + n] = best;
                chain_states[(int64_t)b * (s + 1) + n + 1] = state;
                if (chain_stacks) chain_stacks[(int64_t)b * (s + 1) + n + 1] = encode_stack(&st);
                n++;
                break;
            }
            stack_t_ next = st;
            int32_t end = 0;
            if (!walk_token(p, state, &next, best, &end, NULL)) break;
            proposals[(int64_t)b * s + n] = best;
            state = end;
            st = next;
            n++;
            chain_states[(int64_t)b * (s + 1) + n] = state;
            if (chain_stacks) chain_stacks[(int64_t)b * (s + 1) + n] = encode_stack(&st);
        }
        n_prop[b] = n;
        chain_states[(int64_t)b * (s + 1)] = states[b];
        if (chain_stacks) chain_stacks[(int64_t)b * (s + 1)] = word;
        for (int32_t i = n; i < s; i++) proposals[(int64_t)b * s + i] = -1;
        for (int32_t i = n + 1; i <= s; i++) {
            chain_states[(int64_t)b * (s + 1) + i] = chain_states[(int64_t)b * (s + 1) + n];
            if (chain_stacks) chain_stacks[(int64_t)b * (s + 1) + i] = chain_stacks[(int64_t)b * (s + 1) + n];
        }
    }
}

void oracle_spec_accept(const int32_t* proposals, const int32_t* n_prop, const int32_t* decoded, int32_t batch,
                        int32_t s, int32_t* n_accept) {
    for (int32_t b = 0; b < batch; b++) {
        int32_t k = 0;
        while (k < n_prop[b] && decoded[(int64_t)b * (s + 1) + k] == proposals[(int64_t)b * s + k]) k++;
        n_accept[b] = k;
    }
}

int64_t oracle_advance(const oracle_problem* p, const int32_t* states, const uint64_t* stacks,
                       const int32_t* tokens, int32_t batch, int32_t start_state, int32_t* states_out,
                       uint64_t* stacks_out) {
    int64_t invalid = 0;
    for (int32_t b = 0; b < batch; b++) {
        int32_t t = tokens[b];
        int32_t s = states[b];
        uint64_t w = stacks ? stacks[b] : 0;
        int32_t s_out = 0;
        uint64_t w_out = 0;
        if (t < 0 || t == p->eos_id) {            /* sequence ended: next one starts at init */
            s_out = start_state;
        } else {
            stack_t_ st;
            if (t >= p->n_tokens || !config_valid(p, s, w, &st)) {
                invalid++;
            } else {
                int32_t end = 0;
                if (walk_token(p, s, &st, t, &end, NULL)) {
                    s_out = end;
                    w_out = encode_stack(&st);
                }
            }
        }
        states_out[b] = s_out;
        if (stacks_out) stacks_out[b] = w_out;
    }
    return invalid;
}
