// kernels.cu -- sm_103a kernels of the per-decode-step hot path.
//
//  step_kernel      C.mask() at k = infinity (Alg. 1; Sec. 3.5): every
//                   (sequence, token) pair walks the token's byte classes
//                   through the scanner table (and the bracket stack,
//                   Sec. 3.4) with early exit on the dead state.  One CTA owns
//                   one 1024-token vocabulary window (tokens kept in registers)
//                   and a range of rows; the allowed bits are scattered from
//                   prefix-sorted slot order to original ids in a
//                   shared-memory tile and written out coalesced.  The same
//                   kernel with row = state builds the state x token table
//                   (Alg. 2's traversal, precomputed offline, Sec. 3.5).
//  logits kernels   Alg. 1's v' = m (.) v and greedy decode: one streaming
//                   pass (16-byte loads, masked vectors skipped) computes the
//                   masked max / lowest-index argmax / sum of exp per chunk;
//                   the last CTA of a row combines the chunks (atomic ticket,
//                   no spinning).  Log-probs need a second pass over the row.
//  advance_kernel   C.update(o): the chosen token's walk.
#include <cuda_runtime.h>

#include <climits>
#include <cstdint>

#include "domino_internal.h"

namespace domino {

namespace {

constexpr int kMaxDevices = 64;
constexpr int kMaskTileBytes = 2 * kRowGroup * 32 * 4;
constexpr int kNextTileBytes = 2 * kRowGroup * kWin * 4;

__device__ __forceinline__ uint32_t head_byte(const uint4& h, int i) {
    uint32_t w = (i < 4) ? h.x : (i < 8) ? h.y : (i < 12) ? h.z : h.w;
    return (w >> (8 * (i & 3))) & 0xFFu;
}

template <bool SMEM, typename T>
__device__ __forceinline__ T tload(const T* p, uint32_t i) {
    if constexpr (SMEM) {
        return p[i];
    } else {
        return __ldg(p + i);
    }
}

// DFA walk from s over the token's class string; 0 when the walk dies.
template <bool SMEM>
__device__ __forceinline__ uint32_t walk_dfa(const uint16_t* __restrict__ t, uint32_t K, uint32_t s, const uint4 h,
                                             int len, const uint8_t* __restrict__ tail) {
#pragma unroll
    for (int i = 0; i < kHeadBytes; ++i) {
        if (i >= len) return s;
        s = tload<SMEM>(t, s * K + head_byte(h, i));
        if (s == 0) return 0;
    }
    for (int i = kHeadBytes; i < len; ++i) {
        s = tload<SMEM>(t, s * K + __ldg(tail + (i - kHeadBytes)));
        if (s == 0) return 0;
    }
    return s;
}

// One pushdown step for table entry e (bits 0..15 next, 16..17 kind, 18 sym,
// 19..31 pop-target triple).  Returns the next state, 0 when rejected.
template <bool SMEM>
__device__ __forceinline__ uint32_t pda_step(uint32_t e, uint32_t& bits, uint32_t& depth, uint32_t max_depth,
                                             const uint16_t* __restrict__ ret) {
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
    return tload<SMEM>(ret, (e >> kRetShift) * 4u + revealed);
}

template <bool SMEM>
__device__ __forceinline__ uint32_t walk_pda(const uint32_t* __restrict__ t, const uint16_t* __restrict__ ret,
                                             uint32_t K, uint32_t s, uint32_t& bits, uint32_t& depth,
                                             uint32_t max_depth, const uint4 h, int len,
                                             const uint8_t* __restrict__ tail) {
#pragma unroll
    for (int i = 0; i < kHeadBytes; ++i) {
        if (i >= len) return s;
        s = pda_step<SMEM>(tload<SMEM>(t, s * K + head_byte(h, i)), bits, depth, max_depth, ret);
        if (s == 0) return 0;
    }
    for (int i = kHeadBytes; i < len; ++i) {
        s = pda_step<SMEM>(tload<SMEM>(t, s * K + __ldg(tail + (i - kHeadBytes))), bits, depth, max_depth, ret);
        if (s == 0) return 0;
    }
    return s;
}

// Row configuration; invalid rows become the dead state and report once.
struct RowCfg {
    uint32_t s, bits, depth;
    bool valid;
};

__device__ __forceinline__ RowCfg read_row(const StepView& v, const int32_t* __restrict__ states,
                                           const uint64_t* __restrict__ stacks, int b, bool report) {
    RowCfg c{0u, 0u, 0u, true};
    const int32_t sv = __ldg(states + b);
    uint32_t eb = 0;
    if (sv < 0 || sv >= v.Q) {
        c.valid = false;
        eb |= DOMINO_DEVERR_BAD_STATE;
    }
    if (stacks) {
        const uint64_t w = __ldg(reinterpret_cast<const unsigned long long*>(stacks) + b);
        const uint32_t depth = (uint32_t)(w >> 32) & 0xFFu;
        const uint32_t bits = (uint32_t)w;
        const bool ok = (w >> 40) == 0 && depth <= (uint32_t)v.max_depth && (depth >= 32u || (bits >> depth) == 0);
        if (!ok) {
            c.valid = false;
            eb |= DOMINO_DEVERR_BAD_STACK;
        }
        c.bits = bits;
        c.depth = depth;
    }
    if (c.valid) {
        c.s = (uint32_t)sv;
    } else {
        c.bits = c.depth = 0;
        if (report) atomicOr(v.err, eb);
    }
    return c;
}

template <bool STACK, bool SMEM, bool NEXT>
__global__ void __launch_bounds__(kStepThreads)
    step_kernel(const StepView v, const int32_t* __restrict__ states, const uint64_t* __restrict__ stacks,
                int32_t batch, int32_t rows_per_cta, int32_t row_is_state, uint32_t* __restrict__ mask,
                int32_t* __restrict__ next) {
    extern __shared__ __align__(16) unsigned char smem[];
    uint32_t* mtile = reinterpret_cast<uint32_t*>(smem);
    int32_t* ntile = reinterpret_cast<int32_t*>(smem + kMaskTileBytes);
    unsigned char* tsm = smem + kMaskTileBytes + (NEXT ? kNextTileBytes : 0);

    const int tid = threadIdx.x;
    const int w = blockIdx.x;
    const int row0 = blockIdx.y * rows_per_cta;
    const int row1 = min(batch, row0 + rows_per_cta);
    if (row0 >= row1) return;   // uniform over the CTA, before any barrier

    const uint32_t K = (uint32_t)v.K;
    const uint16_t* t16 = v.t16;
    const uint32_t* t32 = v.t32;
    const uint16_t* ret = v.ret;
    if constexpr (SMEM) {
        // stage the transition table (and pop targets) in shared memory; the
        // device copies are padded to 16 bytes
        const size_t esz = STACK ? 4 : 2;
        const int n_tab = (int)(((size_t)v.Q * K * esz + 15) / 16);
        const int n_ret = (int)(((size_t)v.n_ret * 8 + 15) / 16);
        const uint4* src = STACK ? reinterpret_cast<const uint4*>(v.t32) : reinterpret_cast<const uint4*>(v.t16);
        uint4* dst = reinterpret_cast<uint4*>(tsm);
        for (int i = tid; i < n_tab; i += kStepThreads) dst[i] = __ldg(src + i);
        const uint4* rsrc = reinterpret_cast<const uint4*>(v.ret);
        for (int i = tid; i < n_ret; i += kStepThreads) dst[n_tab + i] = __ldg(rsrc + i);
        t16 = reinterpret_cast<const uint16_t*>(tsm);
        t32 = reinterpret_cast<const uint32_t*>(tsm);
        ret = reinterpret_cast<const uint16_t*>(tsm + (size_t)n_tab * 16);
    }
    for (int i = tid; i < 2 * kRowGroup * 32; i += kStepThreads) mtile[i] = 0u;

    // this thread's tokens (registers for the whole row range)
    uint4 hd[kSlotsPerThread];
    int ln[kSlotsPerThread], ol[kSlotsPerThread];
    bool eos[kSlotsPerThread];
    const uint8_t* tp[kSlotsPerThread];
#pragma unroll
    for (int j = 0; j < kSlotsPerThread; ++j) {
        const int p = w * kWin + tid + j * kStepThreads;
        const int o = __ldg(v.orig + p);
        ol[j] = o >= 0 ? o - w * kWin : -1;
        eos[j] = o >= 0 && o == v.eos_id;
        ln[j] = __ldg(v.len + p);
        hd[j] = __ldg(v.head + p);
        tp[j] = ln[j] > kHeadBytes ? v.tail + __ldg(v.tail_off + p) : v.tail;
    }
    __syncthreads();

    int buf = 0;
    for (int g = row0; g < row1; g += kRowGroup, buf ^= 1) {
        const int nr = min(kRowGroup, row1 - g);
        uint32_t* mt = mtile + buf * kRowGroup * 32;
        int32_t* nt = ntile + buf * kRowGroup * kWin;
#pragma unroll 1
        for (int r = 0; r < nr; ++r) {
            const int b = g + r;
            RowCfg rc;
            if (row_is_state) {
                rc = RowCfg{(uint32_t)b, 0u, 0u, true};
            } else {
                rc = read_row(v, states, stacks, b, w == 0 && tid == 0);
            }
            const bool eos_ok =
                rc.valid && rc.depth == 0 && ((__ldg(v.accept_bits + (rc.s >> 5)) >> (rc.s & 31u)) & 1u);
#pragma unroll
            for (int j = 0; j < kSlotsPerThread; ++j) {
                if (ol[j] < 0) continue;
                uint32_t s;
                if (ln[j] == 0) {
                    s = (eos[j] && eos_ok) ? rc.s : 0u;
                } else if constexpr (STACK) {
                    uint32_t bits = rc.bits, depth = rc.depth;
                    s = walk_pda<SMEM>(t32, ret, K, rc.s, bits, depth, (uint32_t)v.max_depth, hd[j], ln[j], tp[j]);
                } else {
                    s = walk_dfa<SMEM>(t16, K, rc.s, hd[j], ln[j], tp[j]);
                }
                if (s) atomicOr(&mt[r * 32 + (ol[j] >> 5)], 1u << (ol[j] & 31));
                if constexpr (NEXT) nt[r * kWin + ol[j]] = (int32_t)s;
            }
        }
        __syncthreads();
        // write-out of this buffer (the other buffer is used by the next group;
        // the barrier after that group orders this clear before its reuse)
        for (int i = tid; i < nr * 32; i += kStepThreads) {
            const int r = i >> 5, word = w * 32 + (i & 31);
            if (mask && word < v.W) mask[(size_t)(g + r) * v.W + word] = mt[i];
            mt[i] = 0u;
        }
        if constexpr (NEXT) {
            if (v.V % 4 == 0) {
                const int per_row = min(kWin, v.V - w * kWin) / 4;
                for (int i = tid; i < nr * (kWin / 4); i += kStepThreads) {
                    const int r = i / (kWin / 4), k4 = i % (kWin / 4);
                    if (k4 < per_row) {
                        const int4 val = reinterpret_cast<const int4*>(nt + r * kWin)[k4];
                        __stcs(reinterpret_cast<int4*>(next + (size_t)(g + r) * v.V + (size_t)w * kWin) + k4, val);
                    }
                }
            } else {
                for (int i = tid; i < nr * kWin; i += kStepThreads) {
                    const int r = i / kWin, k = i % kWin;
                    const int t = w * kWin + k;
                    if (t < v.V) next[(size_t)(g + r) * v.V + t] = nt[i];
                }
            }
        }
    }
}

// ---------------------------------------------------------------------------
// masked argmax / log-sum-exp
// ---------------------------------------------------------------------------
__device__ __forceinline__ void acc_add(float& m, int& idx, float& s, float x, int t) {
    if (x > m) {
        s = s * __expf(m - x) + 1.0f;
        m = x;
        idx = t;
    } else {
        s += __expf(x - m);
    }
}

// (m, idx, s) <- (m, idx, s) (+) (m2, i2, s2); the larger max wins, the lower
// index on equal maxima; the loser's sum is rescaled to the winner's max.
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
    if (s2 != 0.0f) s += s2 * __expf(m2 - m);
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

template <bool KEEP_L2>
__device__ __forceinline__ uint4 ld_vec(const uint4* p) {
    if constexpr (KEEP_L2) {
        return __ldg(p);
    } else {
        return __ldcs(p);
    }
}

__device__ __forceinline__ uint32_t mask_bits8(const uint32_t* __restrict__ mrow, int v8) {
    return (__ldg(mrow + (v8 >> 2)) >> ((v8 & 3) * 8)) & 0xFFu;
}
__device__ __forceinline__ uint32_t mask_bits4(const uint32_t* __restrict__ mrow, int v4) {
    return (__ldg(mrow + (v4 >> 3)) >> ((v4 & 7) * 4)) & 0xFu;
}
__device__ __forceinline__ bool mask_bit(const uint32_t* __restrict__ mrow, int t) {
    return (__ldg(mrow + (t >> 5)) >> (t & 31)) & 1u;
}

template <bool BF16>
__device__ __forceinline__ float logit_at(const void* row, int t) {
    if constexpr (BF16) {
        const unsigned short u = __ldg(reinterpret_cast<const unsigned short*>(row) + t);
        return __uint_as_float((uint32_t)u << 16);
    } else {
        return __ldg(reinterpret_cast<const float*>(row) + t);
    }
}

constexpr int kUnroll = 4;

template <bool BF16, bool VEC, bool KEEP_L2>
__global__ void __launch_bounds__(kLogitThreads)
    logits_reduce_kernel(const void* __restrict__ logits, int64_t stride, const uint32_t* __restrict__ mask, int V,
                         int W, int chunk, int S, float4* __restrict__ partials, uint32_t* __restrict__ counters,
                         int32_t* __restrict__ argmax, float* __restrict__ lse) {
    const int row = blockIdx.y, c = blockIdx.x, tid = threadIdx.x;
    const int lo = c * chunk, hi = min(V, lo + chunk);
    const uint32_t* mrow = mask + (size_t)row * W;
    const char* lrow = reinterpret_cast<const char*>(logits) + (size_t)row * stride * (BF16 ? 2 : 4);
    float m = -INFINITY, s = 0.0f;
    int idx = INT_MAX;
    int tail_lo = lo;
    if constexpr (VEC) {
        constexpr int E = BF16 ? 8 : 4;   // elements per 16-byte vector
        const int v_lo = lo / E, v_hi = hi / E;
        tail_lo = v_hi * E;
        const uint4* vrow = reinterpret_cast<const uint4*>(lrow);
        for (int v0 = v_lo + tid; v0 < v_hi; v0 += kUnroll * kLogitThreads) {
            uint32_t mb[kUnroll];
            uint4 raw[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int vv = v0 + u * kLogitThreads;
                mb[u] = vv < v_hi ? (BF16 ? mask_bits8(mrow, vv) : mask_bits4(mrow, vv)) : 0u;
                raw[u] = mb[u] ? ld_vec<KEEP_L2>(vrow + vv) : make_uint4(0, 0, 0, 0);
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                if (!mb[u]) continue;
                const int t0 = (v0 + u * kLogitThreads) * E;
                const uint32_t wd[4] = {raw[u].x, raw[u].y, raw[u].z, raw[u].w};
#pragma unroll
                for (int e = 0; e < E; ++e) {
                    if ((mb[u] >> e) & 1u) {
                        float x;
                        if constexpr (BF16) {
                            x = (e & 1) ? bf16_hi(wd[e >> 1]) : bf16_lo(wd[e >> 1]);
                        } else {
                            x = __uint_as_float(wd[e]);
                        }
                        acc_add(m, idx, s, x, t0 + e);
                    }
                }
            }
        }
    }
    for (int t = tail_lo + tid; t < hi; t += kLogitThreads)
        if (mask_bit(mrow, t)) acc_add(m, idx, s, logit_at<BF16>(lrow, t), t);

    // CTA reduction
    __shared__ float sm_m[kLogitThreads / 32], sm_s[kLogitThreads / 32];
    __shared__ int sm_i[kLogitThreads / 32];
    __shared__ int sm_last;
    warp_merge(m, idx, s);
    const int lane = tid & 31, wid = tid >> 5;
    if (lane == 0) {
        sm_m[wid] = m;
        sm_i[wid] = idx;
        sm_s[wid] = s;
    }
    __syncthreads();
    if (wid == 0) {
        m = lane < kLogitThreads / 32 ? sm_m[lane] : -INFINITY;
        idx = lane < kLogitThreads / 32 ? sm_i[lane] : INT_MAX;
        s = lane < kLogitThreads / 32 ? sm_s[lane] : 0.0f;
        warp_merge(m, idx, s);
        if (lane == 0) {
            if (S == 1) {
                argmax[row] = m == -INFINITY ? -1 : idx;
                if (lse) lse[row] = m == -INFINITY ? -INFINITY : m + logf(s);
                sm_last = 0;
            } else {
                partials[(size_t)row * S + c] = make_float4(m, __int_as_float(idx), s, 0.0f);
                __threadfence();
                const unsigned ticket = atomicAdd(counters + row, 1u);
                sm_last = ticket == (unsigned)(S - 1);
            }
        }
    }
    __syncthreads();
    if (sm_last && wid == 0) {
        // last CTA of this row: combine the S chunk partials (S <= 64)
        __threadfence();
        m = -INFINITY;
        s = 0.0f;
        idx = INT_MAX;
        for (int k = lane; k < S; k += 32) {
            const float4 p = __ldcg(partials + (size_t)row * S + k);
            acc_merge(m, idx, s, p.x, __float_as_int(p.y), p.z);
        }
        warp_merge(m, idx, s);
        if (lane == 0) {
            argmax[row] = m == -INFINITY ? -1 : idx;
            if (lse) lse[row] = m == -INFINITY ? -INFINITY : m + logf(s);
            counters[row] = 0u;   // ready for the next launch (stream-ordered)
        }
    }
}

template <bool BF16, bool VEC>
__global__ void __launch_bounds__(kLogitThreads)
    logprobs_kernel(const void* __restrict__ logits, int64_t stride, const uint32_t* __restrict__ mask, int V, int W,
                    int chunk, const float* __restrict__ lse, float* __restrict__ out) {
    const int row = blockIdx.y, c = blockIdx.x, tid = threadIdx.x;
    const int lo = c * chunk, hi = min(V, lo + chunk);
    const uint32_t* mrow = mask + (size_t)row * W;
    const char* lrow = reinterpret_cast<const char*>(logits) + (size_t)row * stride * (BF16 ? 2 : 4);
    float* orow = out + (size_t)row * V;
    const float l = __ldg(lse + row);
    int tail_lo = lo;
    if constexpr (VEC) {
        constexpr int E = BF16 ? 8 : 4;
        const int v_lo = lo / E, v_hi = hi / E;
        tail_lo = v_hi * E;
        const uint4* vrow = reinterpret_cast<const uint4*>(lrow);
        for (int vv = v_lo + tid; vv < v_hi; vv += kLogitThreads) {
            const uint32_t mb = BF16 ? mask_bits8(mrow, vv) : mask_bits4(mrow, vv);
            const uint4 raw = mb ? __ldg(vrow + vv) : make_uint4(0, 0, 0, 0);
            const uint32_t wd[4] = {raw.x, raw.y, raw.z, raw.w};
            float r[E];
#pragma unroll
            for (int e = 0; e < E; ++e) {
                float x;
                if constexpr (BF16) {
                    x = (e & 1) ? bf16_hi(wd[e >> 1]) : bf16_lo(wd[e >> 1]);
                } else {
                    x = __uint_as_float(wd[e]);
                }
                r[e] = ((mb >> e) & 1u) ? x - l : -INFINITY;
            }
            float4* o4 = reinterpret_cast<float4*>(orow + (size_t)vv * E);
            __stcs(o4, make_float4(r[0], r[1], r[2], r[3]));
            if constexpr (BF16) __stcs(o4 + 1, make_float4(r[4], r[5], r[6], r[7]));
        }
    }
    for (int t = tail_lo + tid; t < hi; t += kLogitThreads)
        orow[t] = mask_bit(mrow, t) ? logit_at<BF16>(lrow, t) - l : -INFINITY;
}

// ---------------------------------------------------------------------------
// advance
// ---------------------------------------------------------------------------
template <bool STACK>
__global__ void __launch_bounds__(kAdvanceThreads)
    advance_kernel(const StepView v, const int32_t* __restrict__ states, const uint64_t* __restrict__ stacks,
                   const int32_t* __restrict__ tokens, int32_t batch, int32_t* __restrict__ states_out,
                   uint64_t* __restrict__ stacks_out) {
    const int b = blockIdx.x * kAdvanceThreads + threadIdx.x;
    if (b >= batch) return;
    const int32_t t = tokens[b];
    uint32_t s = 0, bits = 0, depth = 0;
    if (t < 0 || t == v.eos_id) {
        s = (uint32_t)v.start;   // the sequence ended; the next one starts from init
    } else if (t >= v.V) {
        atomicOr(v.err, DOMINO_DEVERR_BAD_TOKEN);
    } else {
        const RowCfg rc = read_row(v, states, stacks, b, true);
        if (rc.valid) {
            const int p = __ldg(v.pos_of + t);
            const int len = __ldg(v.len + p);
            const uint4 h = __ldg(v.head + p);
            const uint8_t* tail = len > kHeadBytes ? v.tail + __ldg(v.tail_off + p) : v.tail;
            if (len > 0) {
                bits = rc.bits;
                depth = rc.depth;
                if constexpr (STACK) {
                    s = walk_pda<false>(v.t32, v.ret, (uint32_t)v.K, rc.s, bits, depth, (uint32_t)v.max_depth, h,
                                        len, tail);
                } else {
                    s = walk_dfa<false>(v.t16, (uint32_t)v.K, rc.s, h, len, tail);
                }
                if (s == 0) bits = depth = 0;
            }
        }
    }
    states_out[b] = (int32_t)s;
    if (stacks_out) stacks_out[b] = ((uint64_t)depth << 32) | bits;
}

template <bool STACK, bool SMEM, bool NEXT>
cudaError_t launch_step_t(const StepView& v, const LaunchEnv& env, const int32_t* states, const uint64_t* stacks,
                          int32_t batch, bool row_is_state, uint32_t* mask, int32_t* next, cudaStream_t st) {
    const int smem = kMaskTileBytes + (NEXT ? kNextTileBytes : 0) + (SMEM ? v.table_bytes : 0);
    auto kern = step_kernel<STACK, SMEM, NEXT>;
    // the dynamic shared-memory limit is raised once per device and size, so
    // that launches inside a stream capture make no attribute calls
    static int configured[kMaxDevices] = {0};
    int dev = 0;
    cudaGetDevice(&dev);
    if (smem > 48 * 1024 && dev < kMaxDevices && configured[dev] < smem) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        configured[dev] = smem;
    }
    const int row_groups = (batch + kRowGroup - 1) / kRowGroup;
    int chunks = (4 * env.num_sms + v.n_windows - 1) / v.n_windows;
    chunks = max(1, min(chunks, row_groups));
    const int rows_per_cta = ((row_groups + chunks - 1) / chunks) * kRowGroup;
    chunks = (batch + rows_per_cta - 1) / rows_per_cta;
    dim3 grid((unsigned)v.n_windows, (unsigned)chunks);
    kern<<<grid, kStepThreads, smem, st>>>(v, states, stacks, batch, rows_per_cta, row_is_state ? 1 : 0, mask,
                                           next);
    return cudaGetLastError();
}

template <bool STACK, bool SMEM>
cudaError_t launch_step_n(const StepView& v, const LaunchEnv& env, const int32_t* states, const uint64_t* stacks,
                          int32_t batch, bool row_is_state, uint32_t* mask, int32_t* next, cudaStream_t st) {
    if (next) return launch_step_t<STACK, SMEM, true>(v, env, states, stacks, batch, row_is_state, mask, next, st);
    return launch_step_t<STACK, SMEM, false>(v, env, states, stacks, batch, row_is_state, mask, next, st);
}

template <bool BF16, bool VEC>
cudaError_t launch_logits_t(const LaunchEnv& env, const void* logits, int32_t batch, int64_t stride, int32_t V,
                            const uint32_t* mask, int32_t* argmax, float* lse, float* logprobs, float4* partials,
                            uint32_t* counters, float* lse_tmp, cudaStream_t st) {
    const int W = (V + 31) / 32;
    const size_t esz = BF16 ? 2 : 4;
    for (int32_t r0 = 0; r0 < batch; r0 += kMaxLogitRows) {
        const int rows = min(kMaxLogitRows, batch - r0);
        int S = (8 * env.num_sms + rows - 1) / rows;
        S = max(1, min(S, min(kMaxChunks, (V + 2047) / 2048)));
        const int chunk = (((V + S - 1) / S) + 7) / 8 * 8;
        S = (V + chunk - 1) / chunk;
        const void* lg = reinterpret_cast<const char*>(logits) + (size_t)r0 * stride * esz;
        const uint32_t* mk = mask + (size_t)r0 * W;
        float* lse_rows = lse ? lse + r0 : (logprobs ? lse_tmp : nullptr);
        dim3 grid((unsigned)S, (unsigned)rows);
        if (logprobs) {
            logits_reduce_kernel<BF16, VEC, true><<<grid, kLogitThreads, 0, st>>>(lg, stride, mk, V, W, chunk, S,
                                                                                  partials, counters, argmax + r0,
                                                                                  lse_rows);
            logprobs_kernel<BF16, VEC><<<grid, kLogitThreads, 0, st>>>(lg, stride, mk, V, W, chunk, lse_rows,
                                                                       logprobs + (size_t)r0 * V);
        } else {
            logits_reduce_kernel<BF16, VEC, false><<<grid, kLogitThreads, 0, st>>>(lg, stride, mk, V, W, chunk, S,
                                                                                   partials, counters, argmax + r0,
                                                                                   lse_rows);
        }
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace

int step_tile_smem_bytes(bool next) { return kMaskTileBytes + (next ? kNextTileBytes : 0); }

cudaError_t launch_step_mask(const StepView& v, const LaunchEnv& env, bool stack, bool smem_table,
                             const int32_t* states, const uint64_t* stacks, int32_t batch, bool row_is_state,
                             uint32_t* mask, int32_t* next, cudaStream_t st) {
    if (stack) {
        if (smem_table) return launch_step_n<true, true>(v, env, states, stacks, batch, row_is_state, mask, next, st);
        return launch_step_n<true, false>(v, env, states, stacks, batch, row_is_state, mask, next, st);
    }
    if (smem_table) return launch_step_n<false, true>(v, env, states, stacks, batch, row_is_state, mask, next, st);
    return launch_step_n<false, false>(v, env, states, stacks, batch, row_is_state, mask, next, st);
}

cudaError_t launch_mask_logits(const LaunchEnv& env, const void* logits, int dtype, int32_t batch,
                               int64_t row_stride, int32_t V, const uint32_t* mask, int32_t* argmax, float* lse,
                               float* logprobs, float4* partials, uint32_t* counters, float* lse_tmp,
                               cudaStream_t st) {
    const bool bf16 = dtype == DOMINO_DTYPE_BF16;
    const size_t esz = bf16 ? 2 : 4;
    bool vec = (reinterpret_cast<uintptr_t>(logits) % 16 == 0) && ((size_t)row_stride * esz) % 16 == 0;
    if (logprobs) vec = vec && (reinterpret_cast<uintptr_t>(logprobs) % 16 == 0) && (V % 4 == 0);
    if (bf16) {
        if (vec)
            return launch_logits_t<true, true>(env, logits, batch, row_stride, V, mask, argmax, lse, logprobs,
                                               partials, counters, lse_tmp, st);
        return launch_logits_t<true, false>(env, logits, batch, row_stride, V, mask, argmax, lse, logprobs, partials,
                                            counters, lse_tmp, st);
    }
    if (vec)
        return launch_logits_t<false, true>(env, logits, batch, row_stride, V, mask, argmax, lse, logprobs, partials,
                                            counters, lse_tmp, st);
    return launch_logits_t<false, false>(env, logits, batch, row_stride, V, mask, argmax, lse, logprobs, partials,
                                         counters, lse_tmp, st);
}

cudaError_t launch_advance(const StepView& v, bool stack, const int32_t* states, const uint64_t* stacks,
                           const int32_t* tokens, int32_t batch, int32_t* states_out, uint64_t* stacks_out,
                           cudaStream_t st) {
    const unsigned grid = (unsigned)((batch + kAdvanceThreads - 1) / kAdvanceThreads);
    if (stack)
        advance_kernel<true><<<grid, kAdvanceThreads, 0, st>>>(v, states, stacks, tokens, batch, states_out,
                                                               stacks_out);
    else
        advance_kernel<false><<<grid, kAdvanceThreads, 0, st>>>(v, states, stacks, tokens, batch, states_out,
                                                                stacks_out);
    return cudaGetLastError();
}

}  // namespace domino
