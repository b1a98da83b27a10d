// walk_common.cuh -- device helpers shared by the kernels of kernels.cu and
// trie.cu: launches with programmatic dependent launch, the online (max,
// lowest-index argmax, sum of exp) fold, the transition table lookups of the
// four table modes, the bracket-stack step, the row configuration decode and
// the update of one row (Alg. 1's update).
#pragma once
#include <cuda_runtime.h>

#include <climits>
#include <cstdint>
#include <type_traits>
#include <utility>

#include "domino_internal.h"

namespace domino {
namespace {

constexpr float kLog2e = 1.4426950408889634f;   // log2(e): exp(x) = 2^(x log2 e)

__host__ __device__ constexpr int align16(int x) { return (x + 15) & ~15; }

// Programmatic dependent launch: a kernel may start while the previous kernel
// of its stream drains; it runs only work that reads nothing the earlier
// kernels write, then waits for them (griddepcontrol.wait returns at once when
// the kernel was launched without the attribute).  Each kernel lets its
// successor launch only after its own wait, so a chain of launches never runs
// more than one kernel ahead.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory"); }

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// A compacted list of the rows to process (opportunistic masking's rejected
// rows): entry i of the pass is row ids[i] of the batch, and only the first
// *count - base entries of this pass exist (the count is device memory).
struct RowList {
    const int32_t* ids;     // nullptr: rows are 0..B-1
    const int32_t* count;
    int32_t base;           // first list entry of this pass
    __device__ __forceinline__ int rows(int cap) const {
        if (!ids) return cap;
        return max(0, min(cap, __ldg(count) - base));
    }
    __device__ __forceinline__ int row(int i) const { return ids ? __ldg(ids + base + i) : i; }
};

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// (m, idx, s) <- (m, idx, s) (+) (m2, i2, s2): larger max wins, lower index on
// equal maxima; the other sum is rescaled to the winner's max.
__device__ __forceinline__ void acc_merge(float& m, int& idx, float& s, float m2, int i2, float s2) {
    if (m2 > m || (m2 == m && i2 < idx)) {
        const float tm = m, ts = s;
        const int ti = idx;
        m = m2;
        idx = i2;
        s = s2;
        m2 = tm;
        i2 = ti;
        s2 = ts;
    }
    if (s2 != 0.0f) s += s2 * ex2((m2 - m) * kLog2e);
}

// one allowed logit x at index t; mL = m * log2(e) is kept with m
__device__ __forceinline__ void acc_add(float& m, float& mL, int& idx, float& s, float x, int t) {
    if (x > m) {
        const float xL = x * kLog2e;
        s = s * ex2(mL - xL) + 1.0f;
        m = x;
        mL = xL;
        idx = t;
    } else {
        s += ex2(fmaf(x, kLog2e, -mL));
    }
}

__device__ __forceinline__ void warp_merge(float& m, int& idx, float& s) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
        const int i2 = __shfl_xor_sync(0xffffffffu, idx, off);
        const float s2 = __shfl_xor_sync(0xffffffffu, s, off);
        acc_merge(m, idx, s, m2, i2, s2);
    }
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// Transition lookup for the four table modes.
template <typename E, int MODE>
struct Tab {
    const E* dense;
    const uint32_t* sp;
    const E* tgt;
    uint32_t K;
#ifdef DOMINO_DEBUG
    // the debug build's bounds (set by debug_bounds): a lookup outside the
    // table sets DOMINO_DEVERR_INTERNAL and reads as the dead state
    uint32_t Q = 0xFFFFFFFFu, nnz = 0xFFFFFFFFu;
    uint32_t* err = nullptr;
    __device__ __forceinline__ bool out_of_bounds(uint32_t s, uint32_t c) const {
        if (s < Q && c < K) return false;
        if (err) atomicOr(err, DOMINO_DEVERR_INTERNAL);
        return true;
    }
    __device__ __forceinline__ bool bad_entry(uint32_t i) const {
        if (i < nnz) return false;
        if (err) atomicOr(err, DOMINO_DEVERR_INTERNAL);
        return true;
    }
#endif
    __device__ __forceinline__ uint32_t get(uint32_t s, uint32_t c) const {
#ifdef DOMINO_DEBUG
        if (out_of_bounds(s, c)) return 0u;
#endif
        if constexpr (MODE == kDenseSmem) {
            return dense[s * K + c];
        } else if constexpr (MODE == kDenseGlobal) {
            return __ldg(dense + s * K + c);
        } else if constexpr (MODE == kSparse32Smem) {
            const uint2 ri = reinterpret_cast<const uint2*>(sp)[s];
            if (!((ri.x >> c) & 1u)) return 0u;
#ifdef DOMINO_DEBUG
            if (bad_entry(ri.y + __popc(ri.x & ((1u << c) - 1u)))) return 0u;
#endif
            return tgt[ri.y + __popc(ri.x & ((1u << c) - 1u))];
        } else {
            const uint4 ri = reinterpret_cast<const uint4*>(sp)[s];
            const unsigned long long m = ((unsigned long long)ri.y << 32) | ri.x;
            if (!((m >> c) & 1ull)) return 0u;
#ifdef DOMINO_DEBUG
            if (bad_entry(ri.z + (uint32_t)__popcll(m & ((1ull << c) - 1ull)))) return 0u;
#endif
            return tgt[ri.z + __popcll(m & ((1ull << c) - 1ull))];
        }
    }
};

// The debug build's table bounds for tab (a no-op otherwise).
template <typename T>
__device__ __forceinline__ void debug_bounds(T& tab, const StepView& v) {
#ifdef DOMINO_DEBUG
    tab.Q = (uint32_t)v.Q;
    tab.nnz = v.sp_nnz > 0 ? (uint32_t)v.sp_nnz : 0xFFFFFFFFu;
    tab.err = v.err;
#else
    (void)tab;
    (void)v;
#endif
}

// One pushdown step for table entry e (bits 0..15 next, 16..17 kind, 18 sym,
// 19..31 pop-target triple).  Returns the next state, 0 when rejected.
__device__ __forceinline__ uint32_t pda_apply(uint32_t e, uint32_t& bits, uint32_t& depth, uint32_t max_depth,
                                              const uint16_t* ret) {
    const uint32_t kind = (e >> kKindShift) & 3u;
    if (kind == 0) return e & 0xFFFFu;
    const uint32_t sym = (e >> kSymShift) & 1u;
    if (kind == 1) {
        if (depth >= max_depth) return 0;
        bits = (bits << 1) | sym;
        ++depth;
        return e & 0xFFFFu;
    }
    if (depth == 0 || (bits & 1u) != sym) return 0;
    bits >>= 1;
    --depth;
    const uint32_t revealed = depth == 0 ? 0u : 1u + (bits & 1u);
    return ret[(e >> kRetShift) * 4u + revealed];
}

// One transition step (with the bracket rules for a pushdown table).
template <bool STACK, typename T>
__device__ __forceinline__ uint32_t step_once(const T& tab, const uint16_t* ret, uint32_t max_depth, uint32_t s,
                                              uint32_t c, uint32_t& bits, uint32_t& depth) {
    const uint32_t e = tab.get(s, c);
    if constexpr (STACK) {
        return pda_apply(e, bits, depth, max_depth, ret);
    } else {
        return e;
    }
}

// Walk bytes FROM..len-1 of a token from state s; 0 when the walk dies.  The
// first 32 class ids are at `head` (shared or global memory), bytes 32.. are in
// `tail` (global memory, touched only by tokens that long).
template <bool STACK, int FROM, typename T>
__device__ __forceinline__ uint32_t walk(const T& tab, const uint16_t* ret, uint32_t max_depth, uint32_t s,
                                         uint32_t& bits, uint32_t& depth, const uint8_t* head, int len,
                                         const uint8_t* __restrict__ tail) {
    const int n1 = min(len, kInlineBytes);
#pragma unroll 1
    for (int i = FROM; i < n1; ++i) {
        s = step_once<STACK>(tab, ret, max_depth, s, head[i], bits, depth);
        if (s == 0) return 0;
    }
#pragma unroll 1
    for (int i = kInlineBytes; i < len; ++i) {
        s = step_once<STACK>(tab, ret, max_depth, s, __ldg(tail + (i - kInlineBytes)), bits, depth);
        if (s == 0) return 0;
    }
    return s;
}

template <bool STACK, int NW, typename T>
__device__ __forceinline__ uint32_t chains_step(const T& tab, const uint16_t* ret, uint32_t max_depth,
                                                uint32_t (&s)[NW], uint32_t (&bits)[NW], uint32_t (&depth)[NW],
                                                uint32_t c) {
    uint32_t alive = 0;
#pragma unroll
    for (int k = 0; k < NW; ++k) {
        s[k] = step_once<STACK>(tab, ret, max_depth, s[k], c, bits[k], depth[k]);
        alive |= s[k];
    }
    return alive;
}

// NW independent walks of one token (bytes 1..len-1) from NW configurations;
// a chain that dies stays 0 (row 0 of every table image is all zero).  `head`
// is the token's first 32 class ids in shared memory.
template <bool STACK, int NW, typename T>
__device__ __forceinline__ void walk_chains(const T& tab, const uint16_t* ret, uint32_t max_depth,
                                            uint32_t (&s)[NW], uint32_t (&bits)[NW], uint32_t (&depth)[NW],
                                            const uint8_t* head, int len, const uint8_t* __restrict__ tail) {
    const int n1 = min(len, kInlineBytes);
#pragma unroll 1
    for (int i = 1; i < n1; ++i)
        if (!chains_step<STACK, NW>(tab, ret, max_depth, s, bits, depth, head[i])) return;
#pragma unroll 1
    for (int i = kInlineBytes; i < len; ++i)
        if (!chains_step<STACK, NW>(tab, ret, max_depth, s, bits, depth, __ldg(tail + (i - kInlineBytes)))) return;
}

// Row configuration: x state, y stack bits, z depth, w flags (1 valid, 2 EOS allowed).
// `sv` / `w` are the raw state and stack word of the row; accept bits may be
// in shared or global memory.
__device__ __forceinline__ uint4 decode_row(const StepView& v, int32_t sv, unsigned long long w, bool has_stack,
                                            const uint32_t* accept_bits, bool report) {
    uint32_t s = 0, bits = 0, depth = 0;
    bool valid = true;
    uint32_t eb = 0;
    if (sv < 0 || sv >= v.Q) {
        valid = false;
        eb |= DOMINO_DEVERR_BAD_STATE;
    }
    if (has_stack) {
        depth = (uint32_t)(w >> 32) & 0xFFu;
        bits = (uint32_t)w;
        const bool ok = (w >> 40) == 0 && depth <= (uint32_t)v.max_depth && (depth >= 32u || (bits >> depth) == 0);
        if (!ok) {
            valid = false;
            eb |= DOMINO_DEVERR_BAD_STACK;
        }
    }
    if (valid) {
        s = (uint32_t)sv;
    } else {
        bits = depth = 0;
        if (report) atomicOr(v.err, eb);
    }
    const bool eos_ok = valid && depth == 0 && ((accept_bits[s >> 5] >> (s & 31u)) & 1u);
    return make_uint4(s, bits, depth, (valid ? 1u : 0u) | (eos_ok ? 2u : 0u));
}

__device__ __forceinline__ uint4 read_row(const StepView& v, const int32_t* __restrict__ states,
                                          const uint64_t* __restrict__ stacks, int b, bool report) {
    const int32_t sv = __ldg(states + b);
    const unsigned long long w = stacks ? __ldg(reinterpret_cast<const unsigned long long*>(stacks) + b) : 0ull;
    return decode_row(v, sv, w, stacks != nullptr, v.accept_bits, report);
}

// read_row for configurations that the same kernel overwrites (the update
// writes its outputs in place): coherent loads, no read-only path.
__device__ __forceinline__ uint4 read_row_rw(const StepView& v, const int32_t* states, const uint64_t* stacks, int b,
                                             bool report) {
    const int32_t sv = __ldcg(states + b);
    const unsigned long long w = stacks ? __ldcg(reinterpret_cast<const unsigned long long*>(stacks) + b) : 0ull;
    return decode_row(v, sv, w, stacks != nullptr, v.accept_bits, report);
}

// C.update() for one row: row b's configuration walks token t (t < 0 or EOS:
// the start state; a rejected token: state 0; t >= V: state 0 and the error
// word).  Reads the configuration before writing, so the outputs may alias it.
template <bool STACK, typename TabT>
__device__ __forceinline__ void advance_row_with(const StepView& v, const TabT& tab, const uint16_t* ret,
                                                 const int32_t* states, const uint64_t* stacks, int b, int32_t t,
                                                 int32_t* states_out, uint64_t* stacks_out) {
    uint32_t s = 0, bits = 0, depth = 0;
    if (t < 0 || t == v.eos_id) {
        s = (uint32_t)v.start;   // the sequence ended; the next one starts from init
    } else if (t >= v.V) {
        atomicOr(v.err, DOMINO_DEVERR_BAD_TOKEN);
    } else {
        const uint4 rc = read_row_rw(v, states, stacks, b, true);
        if (rc.w & 1u) {
            const int p = __ldg(v.pos_of + t);
            const int len = (int)(__ldg(v.info + p) >> 16);
            const uint8_t* hp = reinterpret_cast<const uint8_t*>(v.head + 2 * (size_t)p);
            const uint8_t* tail = len > kInlineBytes ? v.tail + __ldg(v.tail_off + p) : v.tail;
            if (len > 0) {
                bits = rc.y;
                depth = rc.z;
                s = walk<STACK, 0>(tab, ret, (uint32_t)v.max_depth, rc.x, bits, depth, hp, len, tail);
                if (s == 0) bits = depth = 0;
            }
        }
    }
    states_out[b] = (int32_t)s;
    if (stacks_out) stacks_out[b] = ((uint64_t)depth << 32) | bits;
}

// advance_row_with over the table image the step kernel stages, read from
// global memory (L2-resident)
template <bool STACK, int MODE>
__device__ __forceinline__ void advance_row(const StepView& v, const int32_t* states, const uint64_t* stacks, int b,
                                            int32_t t, int32_t* states_out, uint64_t* stacks_out) {
    using E = typename std::conditional<STACK, uint32_t, uint16_t>::type;
    Tab<E, MODE == kDenseSmem ? kDenseGlobal : MODE> tab;
    tab.dense = reinterpret_cast<const E*>(STACK ? (const void*)v.t32 : (const void*)v.t16);
    tab.sp = v.sp_info;
    tab.tgt = reinterpret_cast<const E*>(v.sp_tgt);
    tab.K = (uint32_t)v.K;
    debug_bounds(tab, v);
    advance_row_with<STACK>(v, tab, v.ret, states, stacks, b, t, states_out, stacks_out);
}
}  // namespace
}  // namespace domino
