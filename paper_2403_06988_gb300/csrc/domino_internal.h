// domino_internal.h -- shared between the host-side C ABI (host.cpp) and the
// sm_103a kernels (kernels.cu).  Not part of the public ABI.
#pragma once
#include <cuda_runtime.h>

#include <cstdint>
#include <vector>

#include "domino.h"

namespace domino {

// Vocabulary windows: original ids [w*kWin, (w+1)*kWin) form window w.  Inside
// a window the tokens are stored sorted by their byte-class strings, so that a
// warp walks tokens with common prefixes (same first transitions, same early
// exit) and the mask bits are scattered back to original ids in shared memory.
constexpr int kWin = 1024;
constexpr int kStepThreads = 256;              // step kernel CTA size
constexpr int kSlotsPerThread = kWin / kStepThreads;
constexpr int kRowGroup = 8;                   // rows walked between two write-outs
constexpr int kHeadBytes = 16;                 // class ids stored inline per token
constexpr int kLogitThreads = 256;
constexpr int kMaxLogitRows = 4096;            // rows per mask_logits pass (scratch size)
constexpr int kMaxChunks = 64;                 // CTAs per row in mask_logits
constexpr int kAdvanceThreads = 128;

// Table entry of a pushdown automaton (uint32): bits 0..15 next state, bits
// 16..17 kind (0 none, 1 push, 2 pop), bit 18 symbol, bits 19..31 index of the
// pop's (empty, top0, top1) target triple.  A plain DFA uses uint16 entries.
constexpr uint32_t kKindShift = 16, kSymShift = 18, kRetShift = 19;
constexpr uint32_t kMaxRetTriples = 1u << 13;

struct StepView {
    // vocabulary arena (slot order)
    const uint4* head;        // [n_slots] first 16 class ids
    const int32_t* orig;      // [n_slots] original id, -1 for padding slots
    const uint16_t* len;      // [n_slots] byte length (0 for EOS)
    const int32_t* tail_off;  // [n_slots] offset of bytes 16.. in `tail`
    const uint8_t* tail;      // class ids of bytes 16.. of long tokens
    const int32_t* pos_of;    // [V] slot of original id
    int32_t V, W, n_windows, eos_id;
    // automaton
    const uint16_t* t16;      // [Q][K] (DFA)
    const uint32_t* t32;      // [Q][K] (pushdown)
    const uint16_t* ret;      // [n_ret][4]
    const uint32_t* accept_bits;
    int32_t Q, K, start, max_depth, n_ret;
    int32_t table_bytes;      // bytes of t16/t32 (+ ret) as staged in shared memory
    uint32_t* err;            // sticky device error word
};

struct LaunchEnv {
    int num_sms;
    int max_smem_optin;
};

cudaError_t launch_step_mask(const StepView& v, const LaunchEnv& env, bool stack, bool smem_table,
                             const int32_t* states, const uint64_t* stacks, int32_t batch, bool row_is_state,
                             uint32_t* mask, int32_t* next, cudaStream_t st);

// Shared-memory bytes the step kernel needs for its tiles (without the table).
int step_tile_smem_bytes(bool next);

cudaError_t launch_mask_logits(const LaunchEnv& env, const void* logits, int dtype, int32_t batch,
                               int64_t row_stride, int32_t V, const uint32_t* mask, int32_t* argmax, float* lse,
                               float* logprobs, float4* partials, uint32_t* counters, float* lse_tmp,
                               cudaStream_t st);

cudaError_t launch_advance(const StepView& v, bool stack, const int32_t* states, const uint64_t* stacks,
                           const int32_t* tokens, int32_t batch, int32_t* states_out, uint64_t* stacks_out,
                           cudaStream_t st);

}  // namespace domino
