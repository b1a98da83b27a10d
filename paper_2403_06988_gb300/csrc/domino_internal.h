// domino_internal.h -- shared between the host-side C ABI (host.cpp) and the
// sm_103a kernels (kernels.cu).  Not part of the public ABI.
#pragma once
#include <cuda_runtime.h>

#include <cstdint>
#include <vector>

#include "domino.h"

namespace domino {

// Vocabulary windows: original ids [w*kWin, (w+1)*kWin) form window w.  Inside
// a window the tokens are stored sorted by their byte-class strings, so tokens
// with the same first class form one contiguous group and neighbouring tokens
// share prefixes (same transitions, same early exit for a warp).  The allowed
// bits are scattered back to original ids in shared memory.
constexpr int kWin = 1024;
constexpr int kStepThreads = 1024;             // step kernel CTA size (one CTA per SM)
constexpr int kRowsPerTile = 4;                // fewest rows per tile (mask only; small batches)
constexpr int kMaxRowsPerTile = 32;            // most rows per tile (one warp ballot)
constexpr int kRowsPerTileNext = 8;            // rows per tile when next states are written
constexpr int kWalkChains = 4;                 // rows walked together by one lane (independent chains)
constexpr int kHeadBytes = 16;                 // class ids per 16-byte head block
constexpr int kInlineBytes = 32;               // class ids stored inline per token (two head blocks)
constexpr int kLogitThreads = 256;
constexpr int kMaxLogitRows = 4096;            // rows per mask_logits pass (scratch size)
constexpr int kMaxSegments = 64;               // CTAs sharing one row in mask_logits
constexpr int kAdvanceThreads = 128;

// slot info word: bits 0..9 original id within the window, bit 10 valid,
// bits 16..31 byte length (0 for EOS and empty tokens)
constexpr uint32_t kInfoValid = 1u << 10;

// Table entry of a pushdown automaton (uint32): bits 0..15 next state, bits
// 16..17 kind (0 none, 1 push, 2 pop), bit 18 symbol, bits 19..31 index of the
// pop's (empty, top0, top1) target triple.  A plain DFA uses uint16 entries.
constexpr uint32_t kKindShift = 16, kSymShift = 18, kRetShift = 19;
constexpr uint32_t kMaxRetTriples = 1u << 13;

// Where the step kernel reads transitions from.
enum TableMode : int {
    kDenseSmem = 0,    // [Q][K] entries staged in shared memory
    kSparse32Smem = 1, // per state {live-class mask, base} + packed live entries (K <= 32)
    kSparse64Smem = 2, // the same with a 64-bit class mask (K <= 64)
    kDenseGlobal = 3,  // [Q][K] entries read through L1/L2
};

struct StepView {
    // vocabulary arena (slot order)
    const uint4* head;        // [n_slots][2] class ids of bytes 0..15 and 16..31
    const uint32_t* info;     // [n_slots] original id in window | valid | length
    const int32_t* tail_off;  // [n_slots] offset of bytes 32.. in `tail`
    const uint8_t* tail;      // class ids of bytes 32.. of tokens longer than 32 bytes
    const int32_t* pos_of;    // [V] slot of original id
    // the slots of first class c in window w are [cls_start[w][c], cls_start[w][c + 1])
    const uint16_t* cls_start; // [n_windows][K + 1]
    const int16_t* eos_slot;  // [n_windows] window-local slot of EOS, -1 if not in the window
    int32_t V, W, n_windows, eos_id;
    // automaton
    const uint16_t* t16;      // [Q][K] (DFA)
    const uint32_t* t32;      // [Q][K] (pushdown)
    const uint32_t* sp_info;  // sparse rows: [Q][2] or [Q][4] uint32 words
    const void* sp_tgt;       // sparse live entries (uint16 or uint32)
    const uint16_t* ret;      // [n_ret][4]
    const uint32_t* accept_bits;
    // self loops (nullptr when not used): per state the classes that keep it,
    // per slot the classes of the token's bytes after the first
    const unsigned long long* self_mask;  // [Q]
    const unsigned long long* tok_cls;    // [n_slots]
    int32_t Q, K, start, max_depth, n_ret, sp_nnz;
    uint32_t* err;            // sticky device error word
};

// Prefix tree of the vocabulary's byte-class strings (the subterminal tree of
// Sec. 3.3, Alg. 2, over byte classes): a prefix shared by many tokens takes
// its transitions once per row, and a subtree whose prefix dies is never
// entered.  Nodes are numbered in preorder (children by class), so a subtree
// is the contiguous range [n, skip) and the tokens of a subtree are a
// contiguous range of `dtok`: the tokens that end at n first, then those of
// its children's subtrees.
//   node[2n]     = {skip | cls << 24, tok_lo, n_end, tok_hi}
//   node[2n + 1] = {sub_lo, sub_hi, 0, 0}
// cls: the class on the edge into n; [tok_lo, tok_lo + n_end): tokens ending
// at n; [tok_lo, tok_hi): tokens of the subtree; sub: the classes on the edges
// below n (K <= 64, for the self-loop skip).
// Upper nodes: the root and every node whose subtree has more than kTrieTile
// nodes or more than kTrieBranch branching levels (an ancestor of an upper
// node is upper).  Units: the subtrees hanging off upper nodes.  Inside a
// unit, a node with one child and no token is walked together with its child:
// the walk's records are such runs (up to 255 nodes).  The units are cut into
// per-CTA batches that fit in shared memory; for a block of rows a CTA
// computes each row's configuration at the upper nodes its units hang off
// ("slots"), then each (unit, row live at its slot) pair is walked by one
// thread, depth first over the unit's records, with a stack of at most
// kTrieBranch entries (tree_tile_kernel).  The tokens that end at an upper
// node are set by the one batch that lists that node as an emitting slot.
constexpr int kTrieTile = 64;
constexpr int kTrieBranch = 8;
constexpr int kTrieInterleave = 2;      // places of the tree a CTA's units are drawn from
constexpr int kTrieMaxSlots = 48;             // slots per batch
constexpr int32_t kTrieMaxNodes = (1 << 24) - 1;

struct TrieView {
    const uint4* node;        // the walk's records, two each: {end record, first node, nodes, first token},
                              //   {tokens ending at the last node, classes below it (64 bits), 0}
    const uint8_t* ncls;      // [n_nodes]: each node's class (the records' classes, in order)
    const int32_t* dtok;      // original ids in preorder
    const uint4* upper;       // [n_upper]: {node, path offset, path length, 0}
    const uint8_t* upath;     // classes of the upper nodes' paths from the root
    const uint4* batch;       // [n_batches][2]: {first unit, end unit, first range, end range},
                              //                 {first slot, end slot, staged nodes, staged tokens}
    const uint4* range;       // two each: {first record, end record, first token, end token},
                              //   {first node, end node, 0, 0}; staged one after the other
    const uint4* slot;        // {upper index, first token ending at its node, tokens it sets (0: none), 0}
    const uint2* unit;        // {root's staged index, slot index within the batch}
    const int32_t* cta_batch; // [grid + 1]: CTA c takes batches [cta_batch[c], cta_batch[c + 1])
    int32_t n_nodes, n_upper, grid, n_batches;
    int32_t max_nodes, max_cls, max_toks, max_units, max_slots, max_path;   // the largest batch (records, nodes, ...)
};

struct LaunchEnv {
    int num_sms;
    int max_smem_optin;
};

// Bytes the table of `mode` occupies in shared memory (0 for kDenseGlobal).
int64_t table_smem_bytes(const StepView& v, bool stack, int mode);

// Shared-memory bytes of the step kernel other than the table.
int step_fixed_smem_bytes(const StepView& v, bool next);

// row_ids / row_count (device): only rows row_ids[i], i < *row_count <= batch,
// are walked; their masks are written to the compact rows i of `mask`.
cudaError_t launch_step_mask(const StepView& v, const LaunchEnv& env, bool stack, int mode, const int32_t* states,
                             const uint64_t* stacks, int32_t batch, bool row_is_state, uint32_t* mask,
                             int32_t* next, cudaStream_t st, const int32_t* row_ids = nullptr,
                             const int32_t* row_count = nullptr, const void* fuse_logits = nullptr,
                             int64_t fuse_stride = 0, float4* fuse_part = nullptr, bool fuse_prefetch = false);

// The mask step fused with the masked decode (bf16 logits, rows on 16-byte
// boundaries): fuse_part [batch][n_windows] receives per-window partials,
// merged into argmax / lse by launch_fused_combine, which also advances each
// row by its argmax when states_out is given (outputs may alias the inputs).
cudaError_t launch_fused_combine(const StepView& v, bool stack, int mode, const float4* part, int32_t batch,
                                 int32_t n_windows, int32_t* argmax, float* lse, const int32_t* states,
                                 const uint64_t* stacks, int32_t* states_out, uint64_t* stacks_out, cudaStream_t st);

// The mask step over the prefix tree: tree_clear_kernel (one warp per row:
// clears the row's mask and next states, sets EOS), then tree_tile_kernel
// (the units, from shared memory).  states / stacks / batch / row_is_state /
// mask / next / row_ids / row_count as launch_step_mask.  mode: where the tile
// kernel reads transitions.
int trie_tile_smem_bytes(const StepView& v, const TrieView& tv, bool stack, int table_bytes);
// row_next (the precompute: row_is_state, next states written, no row list):
// tv.n_batches device words through which the CTAs share out the batches' row
// blocks (nullptr: each CTA walks every row of its own batches).
cudaError_t launch_trie_step(const StepView& v, const TrieView& tv, const LaunchEnv& env, bool stack, int mode,
                             const int32_t* states, const uint64_t* stacks, int32_t batch, bool row_is_state,
                             uint32_t* mask, int32_t* next, cudaStream_t st, const int32_t* row_ids = nullptr,
                             const int32_t* row_count = nullptr, int32_t* row_next = nullptr);

// Log-probabilities only (bf16 logits, rows on 16-byte boundaries), given the
// rows' lse: logprobs[b][t] = logit - lse[b] for allowed t, -inf else.
cudaError_t launch_logprobs_bf16(const LaunchEnv& env, const void* logits, int32_t batch, int64_t row_stride,
                                 int32_t V, const uint32_t* mask, const float* lse, float* logprobs, cudaStream_t st);

// Sampling decode: Gumbel-max with Philox4x32-10 uniforms (kernels.cu).
struct SampleArgs {
    uint32_t key0, key1;     // the 64-bit seed
    uint32_t off0, off1;     // the 64-bit offset (counter words 2 and 3)
    float inv_t;             // 1 / temperature, rounded to fp32
};

// row_state (table-driven step): row r's mask is row row_state[r] of the
// [Q][W] table `mask`; out-of-range states read as empty rows and set `err`.
// sample: draw each row's token (into argmax) instead of the greedy argmax;
// lse and logprobs must then be null.  mask == nullptr (no row_state): every
// token allowed.  row_ids / row_count (device): only rows row_ids[i] for
// i < *row_count are processed, their masks being the compact rows i of
// `mask`; argmax and lse are indexed by batch row; no logprobs.
// raises the logits kernels' shared-memory limit on the current device; called
// once per handle and device, outside any stream capture
cudaError_t prepare_logits_kernels();
cudaError_t launch_mask_logits(const LaunchEnv& env, const void* logits, int dtype, int32_t batch,
                               int64_t row_stride, int32_t V, const uint32_t* mask, int32_t* argmax, float* lse,
                               float* logprobs, float4* partials, uint32_t* counters, float* lse_tmp,
                               cudaStream_t st, const int32_t* row_state = nullptr, int32_t Q = 0,
                               uint32_t* err = nullptr, const SampleArgs* sample = nullptr,
                               const int32_t* row_ids = nullptr, const int32_t* row_count = nullptr);

// Fills the sampling arguments (1/T in fp32, seed and offset words).
cudaError_t launch_mask_sample(const LaunchEnv& env, const void* logits, int dtype, int32_t batch,
                               int64_t row_stride, int32_t V, const uint32_t* mask, float temperature,
                               uint64_t seed, uint64_t offset, int32_t* tokens, float4* partials,
                               uint32_t* counters, cudaStream_t st);

// `mode` names the table image the step kernel reads (it is L2-resident after a step).
cudaError_t launch_advance(const StepView& v, bool stack, int mode, const int32_t* states, const uint64_t* stacks,
                           const int32_t* tokens, int32_t batch, int32_t* states_out, uint64_t* stacks_out,
                           cudaStream_t st);

cudaError_t launch_advance_table(const int32_t* table_next, int32_t Q, int32_t V, int32_t eos_id, int32_t start,
                                 const int32_t* states, const int32_t* tokens, int32_t batch, int32_t* states_out,
                                 uint32_t* err, cudaStream_t st);

// Opportunistic masking: accepts row b's proposal into tokens_out[b] or
// appends b to row_ids (counter *row_count, zeroed by the caller).
cudaError_t launch_propose_check(const StepView& v, bool stack, int mode, const int32_t* states,
                                 const uint64_t* stacks, const int32_t* proposals, int32_t batch, int32_t* tokens_out,
                                 int32_t* row_ids, int32_t* row_count, cudaStream_t st);

// Count-based speculation (Sec. 3.6): count update, proposals, acceptance.
cudaError_t launch_spec_update(const StepView& v, bool stack, const int32_t* states, const uint64_t* stacks,
                               const int32_t* tokens, int32_t batch, uint32_t* counts, unsigned long long* best,
                               uint32_t* reached, cudaStream_t st);
cudaError_t launch_spec_propose(const StepView& v, bool stack, int mode, const int32_t* states,
                                const uint64_t* stacks, int32_t batch, int32_t s, int32_t min_permille,
                                const unsigned long long* best, const uint32_t* reached, int32_t* proposals,
                                int32_t* n_prop, int32_t* chain_states, uint64_t* chain_stacks, cudaStream_t st);
cudaError_t launch_spec_accept(const int32_t* proposals, const int32_t* n_prop, const int32_t* decoded,
                               const int32_t* chain_states, const uint64_t* chain_stacks, int32_t batch, int32_t s,
                               int32_t* n_accept, int32_t* tokens_out, int32_t* states_out, uint64_t* stacks_out,
                               cudaStream_t st);


}  // namespace domino
