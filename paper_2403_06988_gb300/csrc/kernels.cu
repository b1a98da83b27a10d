// kernels.cu -- sm_103a kernels of the per-decode-step hot path.
//
//  step_kernel      C.mask() at lookahead k = infinity (Alg. 1; Sec. 3.5):
//                   every (sequence, token) pair walks the token's byte classes
//                   through the scanner table (and the bracket stack,
//                   Sec. 3.4) with early exit on the dead state.  Persistent
//                   CTAs (one per SM) hold the transition table in shared
//                   memory (dense, or sparse per-state live-class masks) and
//                   loop over tiles = (vocabulary window of 1024 tokens,
//                   group of rows).  Inside a window tokens are sorted by
//                   their class strings, so all tokens with the same first
//                   class form one group: per row, the first transition is
//                   taken once per class and only the groups whose first step
//                   is live are walked (work proportional to the surviving
//                   tokens).  Allowed bits are scattered to original ids in a
//                   shared-memory tile and written out coalesced.  The same
//                   kernel with row = state builds the state x token table
//                   (Alg. 2's traversal, precomputed offline, Sec. 3.5), and,
//                   over a device-side row list, masks only the rows that
//                   opportunistic masking rejected.
//  logits_reduce    Alg. 1's v' = m (.) v and decode: a balanced flat split of
//                   the batch x mask words over one-warp CTAs; the 16-byte
//                   logit vectors that hold an allowed token are staged with
//                   cp.async (the others are never read); a lane folds its
//                   word into a masked max / lowest-index argmax / sum of
//                   exp, or a Gumbel-max draw (sampling); per-row segments are
//                   combined by the last CTA to finish (atomic ticket, no
//                   spinning).  Rows may come from a precomputed mask table
//                   (table-driven step) or a device-side row list.
//  logprobs         the second pass for log-probabilities.
//  advance          C.update(o): the chosen token's walk (or one read of the
//                   precomputed next-state table).
//  propose_check,   opportunistic masking's one-walk check, and count-based
//  spec_*           speculation (Sec. 3.6): count update, proposals, acceptance.
#include <cuda_runtime.h>

#include <climits>
#include <cstdint>
#include <mutex>
#include <utility>
#include <algorithm>
#include <type_traits>

#include "domino_internal.h"
#include "walk_common.cuh"

namespace domino {

namespace {

constexpr int kMaxDevices = 64;
static_assert(kStepThreads == kWin, "one thread per window slot");


// The mask step fused with the masked decode: after each tile's walk, warp r
// folds row r's allowed bf16 logits of the tile's window into a (max, argmax,
// sum of exp) partial per (row, window); a combine kernel merges a row's
// windows.  A window with at most 32 allowed tokens lists them one per lane,
// loads their logits and folds them after the next tile's walk; a denser
// window is folded at once, lane j over mask word j.  `logits` may point to
// device memory or to pinned host memory.
__device__ __forceinline__ void prefetch_l2(const void* p) {
    asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

// Folds one row window whose allowed tokens (at most 32) were listed one per
// lane: t = INT_MAX marks an empty lane, raw the lane's bf16 logit.  Writes
// (max, lowest index of the max, sum of exp against the max) to *out.
__device__ __forceinline__ void fold_listed(float4* out, unsigned short raw, int t, int lane) {
    const float x = t != INT_MAX ? __uint_as_float((uint32_t)raw << 16) : -INFINITY;
    float m = x;
    int idx = t;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
        const int i2 = __shfl_xor_sync(0xffffffffu, idx, off);
        if (m2 > m || (m2 == m && i2 < idx)) {
            m = m2;
            idx = i2;
        }
    }
    float e = t != INT_MAX ? ex2(fmaf(x, kLog2e, -m * kLog2e)) : 0.0f;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) e += __shfl_xor_sync(0xffffffffu, e, off);
    if (lane == 0) *out = make_float4(m, __int_as_float(idx), e, 0.f);
}

// The fused masked decode of one row window: `mrow` holds the row's 32 mask
// words of window w in shared memory (the warp owns them and uses them as
// scratch), `lrow` is the row's bf16 logits (device or pinned host memory).
// Writes (max, lowest index of the max, sum of exp against the max) to *out.
// By the number n of allowed tokens: n <= 32 lists them one per lane; n <= 128
// lists them as 16-bit entries and loads up to four per lane at once; denser
// windows are folded word by word, a word's four 16-byte vectors loaded at once.
__device__ __forceinline__ void fold_window(uint32_t* mrow, const char* lrow, int w, int V, int W, int lane,
                                            float4* out) {
    const int full_words = V / 32;
    const int j = w * 32 + lane;
    const uint32_t word = j < W ? mrow[lane] : 0u;
    const unsigned short* u = reinterpret_cast<const unsigned short*>(lrow);
    const int c = __popc(word);
    const int n = __reduce_add_sync(0xffffffffu, c);
    // exclusive offset of the lane's tokens in the row window's list
    // (lane order, then bit order)
    int o = 0;
    if (n <= 128) {
        o = c;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, o, d);
            if (lane >= d) o += y;
        }
        o -= c;
    }
    if (n <= 32) {
        // few allowed tokens: listed one per lane, one logit load per lane
        __syncwarp();
        uint32_t wd = word;
        int oo = o;
        while (wd) {
            const int e = __ffs(wd) - 1;
            wd &= wd - 1;
            mrow[oo++] = (uint32_t)(lane * 32 + e);
        }
        __syncwarp();
        int t = INT_MAX;
        unsigned short raw = 0;
        if (lane < n) {
            t = w * kWin + (int)mrow[lane];
            raw = __ldcs(u + t);
        }
        fold_listed(out, raw, t, lane);
    } else if (n <= 128) {
        // up to four tokens per lane: listed (16-bit entries, two
        // rounds of 64) and loaded together, then a lane-local
        // maximum, the warp's argmax and the warp's sum
        unsigned short* lst = reinterpret_cast<unsigned short*>(mrow);
        int tk[4];
        unsigned short raw[4];
        uint32_t wd = word;
        int oo = o;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            __syncwarp();
            while (wd && oo < 64 * (h + 1)) {
                const int e = __ffs(wd) - 1;
                wd &= wd - 1;
                lst[oo++ - 64 * h] = (unsigned short)(lane * 32 + e);
            }
            __syncwarp();
#pragma unroll
            for (int q = 0; q < 2; ++q) {
                const int k = 64 * h + 32 * q + lane;
                tk[2 * h + q] = k < n ? w * kWin + (int)lst[k - 64 * h] : INT_MAX;
                raw[2 * h + q] = k < n ? __ldcs(u + tk[2 * h + q]) : (unsigned short)0;
            }
        }
        float m = -INFINITY;
        int idx = INT_MAX;
#pragma unroll
        for (int q = 0; q < 4; ++q) {   // tokens ascend with q
            const float x = __uint_as_float((uint32_t)raw[q] << 16);
            if (tk[q] != INT_MAX && x > m) {
                m = x;
                idx = tk[q];
            }
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
            const int i2 = __shfl_xor_sync(0xffffffffu, idx, off);
            if (m2 > m || (m2 == m && i2 < idx)) {
                m = m2;
                idx = i2;
            }
        }
        const float mL = m * kLog2e;
        float sum = 0.0f;
#pragma unroll
        for (int q = 0; q < 4; ++q)
            if (tk[q] != INT_MAX) sum += ex2(fmaf(__uint_as_float((uint32_t)raw[q] << 16), kLog2e, -mL));
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
        if (lane == 0)
            *out = make_float4(m, __int_as_float(idx), sum, 0.f);
    } else {
        float m = -INFINITY, mL = -INFINITY, sum = 0.0f;
        int idx = INT_MAX;
        uint32_t wd = word;
        const int t0 = j * 32;
        if (wd && j < full_words) {
            // many allowed tokens: each lane folds its own word, the
            // word's four 16-byte vectors loaded at once; compact
            // loops, since where masks are sparse this path runs
            // rarely and its code is fetched cold
            const uint4* src = reinterpret_cast<const uint4*>(lrow) + (size_t)j * 4;
            const uint4 z = make_uint4(0u, 0u, 0u, 0u);
            const uint4 q0 = (wd & 0xFFu) ? __ldcs(src) : z;
            const uint4 q1 = (wd & 0xFF00u) ? __ldcs(src + 1) : z;
            const uint4 q2 = (wd & 0xFF0000u) ? __ldcs(src + 2) : z;
            const uint4 q3 = (wd & 0xFF000000u) ? __ldcs(src + 3) : z;
            // the word's maximum (lowest index on ties), then the sum of
            // its terms: no dependence chain through the exponentials
            int wi = 0;
#pragma unroll 1
            for (int k = 0; k < 4; ++k) {
                const uint32_t bits = (wd >> (8 * k)) & 0xFFu;
                const uint4 q = k == 0 ? q0 : k == 1 ? q1 : k == 2 ? q2 : q3;
                const uint32_t qs[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const float x = (e & 1) ? bf16_hi(qs[e >> 1]) : bf16_lo(qs[e >> 1]);
                    if (((bits >> e) & 1u) && x > m) {
                        m = x;
                        wi = 8 * k + e;
                    }
                }
            }
            mL = m * kLog2e;
            idx = t0 + wi;
#pragma unroll 1
            for (int k = 0; k < 4; ++k) {
                const uint32_t bits = (wd >> (8 * k)) & 0xFFu;
                const uint4 q = k == 0 ? q0 : k == 1 ? q1 : k == 2 ? q2 : q3;
                const uint32_t qs[4] = {q.x, q.y, q.z, q.w};
                float acc = 0.0f;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const float x = (e & 1) ? bf16_hi(qs[e >> 1]) : bf16_lo(qs[e >> 1]);
                    acc += ((bits >> e) & 1u) ? ex2(fmaf(x, kLog2e, -mL)) : 0.0f;
                }
                sum += acc;
            }
        } else {   // the row's partial last word
            while (wd) {
                const int e = __ffs(wd) - 1;
                wd &= wd - 1;
                if (t0 + e < V)
                    acc_add(m, mL, idx, sum, __uint_as_float((uint32_t)__ldcs(u + t0 + e) << 16), t0 + e);
            }
        }
        warp_merge(m, idx, sum);
        if (lane == 0)
            *out = make_float4(m, __int_as_float(idx), sum, 0.f);
    }
}

struct FuseArgs {
    const void* logits;   // nullptr: no fusion
    int64_t stride;       // row stride in elements
    float4* part;         // [batch][n_windows] partials
    int prefetch;         // logits in device memory: pull each tile's rows into L2 ahead of the fold
};

// Shared-memory layout of the step kernel (offsets in bytes).
struct StepLayout {
    int head, info, cls, tokcls, pairs, rows, ctrl, cfg, mtile, ntile, accept, self, table, total;
};

// Walk pairs: (token slot, group of up to kWalkChains live rows of the token's
// first class), packed as slot (bits 0..9) | the group's rows (5 bits each,
// bits 10..29) | rows in the group - 1 (bits 30..31).  A tile lists at most
// kWin x ceil(R / kWalkChains) of them.
static_assert(kWalkChains == 4 && kMaxRowsPerTile <= 32 && kWin == 1024, "walk pair packing");

__host__ __device__ inline StepLayout step_layout(int K, int R, bool next, bool stack, int Q, int table_bytes,
                                                  bool self) {
    StepLayout L{};
    int o = 0;
    L.head = o;    o += kWin * 32;
    L.info = o;    o += kWin * 4;
    L.cls = o;     o += align16((K + 1) * 2);
    L.tokcls = o;  o += self ? kWin * 8 : 0;
    L.pairs = o;   o += kWin * ((R + kWalkChains - 1) / kWalkChains) * 4;
    L.rows = o;    o += R * 16;
    L.ctrl = o;    o += 32;
    L.cfg = o;     o += align16(R * K * (stack ? 16 : 4));
    L.mtile = o;   o += align16(R * 32 * 4) * (next ? 1 : 2);   // mask only: two tiles, see step_kernel
    L.ntile = o;   o += next ? R * kWin * 2 : 0;   // next states < Q <= 65535: staged as u16
    L.accept = o;  o += align16(((Q + 31) / 32) * 4);
    L.self = o;    o += self ? align16(Q * 8) : 0;
    L.table = o;   o += align16(table_bytes);
    L.total = o;
    return L;
}

template <bool STACK, int MODE, bool NEXT>
__global__ void __launch_bounds__(kStepThreads, 1)
    step_kernel(const StepView v, const uint4* __restrict__ img, int img_bytes, int img_tgt_off, int img_ret_off,
                const int32_t* __restrict__ states, const uint64_t* __restrict__ stacks, int32_t batch,
                int32_t R, int32_t n_row_tiles, int32_t n_tiles, int32_t row_is_state, uint32_t* __restrict__ mask,
                int32_t* __restrict__ next, const RowList list, const FuseArgs fuse) {
    using E = typename std::conditional<STACK, uint32_t, uint16_t>::type;
    extern __shared__ __align__(16) unsigned char smem[];
    const int K = v.K;
    const bool use_self = v.self_mask != nullptr;
    const StepLayout L = step_layout(K, R, NEXT, STACK, v.Q, MODE == kDenseGlobal ? 0 : img_bytes, use_self);
    uint4* s_head = reinterpret_cast<uint4*>(smem + L.head);
    uint32_t* s_info = reinterpret_cast<uint32_t*>(smem + L.info);
    uint16_t* s_cls = reinterpret_cast<uint16_t*>(smem + L.cls);      // [K + 1] first slot of each first class
    uint32_t* s_pairs = reinterpret_cast<uint32_t*>(smem + L.pairs);   // walk pairs of the tile
    uint4* s_rows = reinterpret_cast<uint4*>(smem + L.rows);
    // rows drained, pairs listed, EOS slot, last rows drained, chunks claimed
    int* s_ctrl = reinterpret_cast<int*>(smem + L.ctrl);
    uint32_t* s_cfg = reinterpret_cast<uint32_t*>(smem + L.cfg);   // [R][K] state (DFA)
    uint4* s_cfg4 = reinterpret_cast<uint4*>(smem + L.cfg);        // [R][K] (state, bits, depth) (pushdown)
    uint32_t* s_mtile = reinterpret_cast<uint32_t*>(smem + L.mtile);
    uint16_t* s_ntile = reinterpret_cast<uint16_t*>(smem + L.ntile);   // [R][kWin] next states
    uint32_t* s_accept = reinterpret_cast<uint32_t*>(smem + L.accept);
    unsigned long long* s_self = reinterpret_cast<unsigned long long*>(smem + L.self);       // [Q]
    unsigned long long* s_tokcls = reinterpret_cast<unsigned long long*>(smem + L.tokcls);   // [kWin]
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (list.ids) {   // a row list may be empty: learn its length before staging anything
        pdl_wait();
        pdl_trigger();
        if (list.rows(batch) == 0) return;
    }
    for (int i = tid; i < (v.Q + 31) / 32; i += kStepThreads) s_accept[i] = __ldg(v.accept_bits + i);
    if (use_self)
        for (int i = tid; i < v.Q; i += kStepThreads) s_self[i] = __ldg(v.self_mask + i);

    Tab<E, MODE> tab;
    tab.K = (uint32_t)K;
    debug_bounds(tab, v);
    const uint16_t* ret;
    if constexpr (MODE == kDenseGlobal) {
        tab.dense = reinterpret_cast<const E*>(STACK ? (const void*)v.t32 : (const void*)v.t16);
        ret = v.ret;
    } else {
        // stage the table image (dense or sparse, plus pop targets) once per CTA
        uint4* dst = reinterpret_cast<uint4*>(smem + L.table);
        for (int i = tid; i < img_bytes / 16; i += kStepThreads) dst[i] = __ldg(img + i);
        const unsigned char* tb = smem + L.table;
        tab.dense = reinterpret_cast<const E*>(tb);
        tab.sp = reinterpret_cast<const uint32_t*>(tb);
        tab.tgt = reinterpret_cast<const E*>(tb + img_tgt_off);
        ret = reinterpret_cast<const uint16_t*>(tb + img_ret_off);
    }
    const uint32_t maxd = (uint32_t)v.max_depth;
    pdl_wait();      // everything below may read what earlier kernels wrote
    pdl_trigger();   // after the wait: at most two kernels of a stream overlap
    if (list.ids) {  // a compacted row list: its length is known only now
        batch = list.rows(batch);
        n_row_tiles = (batch + R - 1) / R;
        n_tiles = n_row_tiles * v.n_windows;
    }

    const int t0 = (int)(((long long)blockIdx.x * n_tiles) / gridDim.x);
    const int t1 = (int)(((long long)(blockIdx.x + 1) * n_tiles) / gridDim.x);
    // the raw configuration of row r0+tid of the coming tile (threads < R),
    // loaded one tile ahead so that its latency overlaps the walk
    int32_t pf_s = 0;
    unsigned long long pf_w = 0ull;
    auto prefetch = [&](int t) {
        if (t < t1 && tid < R && !row_is_state) {
            const int wq = t / n_row_tiles;
            const int b = (t - wq * n_row_tiles) * R + tid;
            if (b < batch) {
                const int rb = list.row(b);
                pf_s = __ldg(states + rb);
                if (stacks) pf_w = __ldg(reinterpret_cast<const unsigned long long*>(stacks) + rb);
            }
        }
    };
    prefetch(t0);
    int cur_w = -1;
    // Mask only (no next states): the mask tile is double-buffered and a
    // tile's write-out and masked decode run in the next tile's walk interval,
    // a row at a time to whichever warp asks next (warps that finish walking
    // early take them); the last tile's after the loop.  pw / pr0 / pnr: the
    // previous tile's window, first row and row count.
    int pw = 0, pr0 = 0, pnr = 0;
    // the previous tile's rows: each warp that asks takes one, writes its 32
    // mask words out, folds its allowed logits (fused decode) and clears the
    // words for the tile after next
    auto drain = [&](int tp, int* counter) {
        uint32_t* pm = s_mtile + (tp & 1) * R * 32;
        for (;;) {
            int r = 0;
            if (lane == 0) r = atomicAdd(counter, 1);
            r = __shfl_sync(0xffffffffu, r, 0);
            if (r >= pnr) break;
            const int j = pw * 32 + lane;
            if (mask && j < v.W) mask[(size_t)(pr0 + r) * v.W + j] = pm[r * 32 + lane];
            if (fuse.logits)
                fold_window(pm + r * 32, reinterpret_cast<const char*>(fuse.logits) + (size_t)(pr0 + r) * fuse.stride * 2,
                            pw, v.V, v.W, lane, fuse.part + (size_t)(pr0 + r) * v.n_windows + pw);
            __syncwarp();
            pm[r * 32 + lane] = 0u;
        }
    };
    if constexpr (!NEXT) {
        for (int i = tid; i < 2 * R * 32; i += kStepThreads) s_mtile[i] = 0u;
        if (tid == 0) s_ctrl[3] = 0;   // the last tile's row counter
    }
    for (int t = t0; t < t1; ++t) {
        const int w = t / n_row_tiles;
        const int r0 = (t - w * n_row_tiles) * R;
        const int nr = min(R, batch - r0);
        uint32_t* mt = s_mtile + (NEXT ? 0 : (t & 1) * R * 32);   // this tile's mask words [R][32]
        __syncthreads();   // the previous tile's walk is done
        if (tid == 0) {
            s_ctrl[0] = 0;   // rows of the previous tile handed out
            s_ctrl[1] = 0;   // pairs listed so far
            s_ctrl[4] = 0;   // chunks of 32 pairs claimed
        }
        if (w != cur_w) {
            s_head[2 * tid] = __ldg(v.head + 2 * ((size_t)w * kWin + tid));
            s_head[2 * tid + 1] = __ldg(v.head + 2 * ((size_t)w * kWin + tid) + 1);
            s_info[tid] = __ldg(v.info + (size_t)w * kWin + tid);
            if (use_self) s_tokcls[tid] = __ldg(v.tok_cls + (size_t)w * kWin + tid);
            for (int i = tid; i <= K; i += kStepThreads) s_cls[i] = __ldg(v.cls_start + (size_t)w * (K + 1) + i);
            if (tid == 0) s_ctrl[2] = __ldg(v.eos_slot + w);
            cur_w = w;
        }
        if (tid < nr) {
            if (row_is_state) {
                const uint32_t q = (uint32_t)(r0 + tid);
                s_rows[tid] = make_uint4(q, 0u, 0u, 1u | (((s_accept[q >> 5] >> (q & 31u)) & 1u) ? 2u : 0u));
            } else {
                s_rows[tid] = decode_row(v, pf_s, pf_w, stacks != nullptr, s_accept, w == 0);
            }
        }
        if constexpr (NEXT)
            for (int i = tid; i < nr * 32; i += kStepThreads) mt[i] = 0u;
        if (fuse.prefetch) {
            // the tile's logits head for L2 while the walk runs: one 128-byte
            // line per thread, every line start inside the row's window slice
            const int win_bytes = min(kWin, v.V - w * kWin) * 2;
            for (int i = tid; i < nr * (kWin * 2 / 128); i += kStepThreads) {
                const int r = i / (kWin * 2 / 128), off = (i % (kWin * 2 / 128)) * 128;
                if (off < win_bytes)
                    prefetch_l2(reinterpret_cast<const char*>(fuse.logits) + (size_t)(r0 + r) * fuse.stride * 2 +
                                (size_t)w * kWin * 2 + off);
            }
        }
        if constexpr (NEXT) {
            for (int i = tid; i < nr * (kWin / 8); i += kStepThreads)
                reinterpret_cast<int4*>(s_ntile)[i] = make_int4(0, 0, 0, 0);
        }
        __syncthreads();

        // first transition once per (row, first class): lane r of a warp takes
        // row r, the ballot gives the class's live rows; the warp then lists
        // the class's walk pairs, every (token, group of up to kWalkChains
        // live rows) with the group's rows packed into the pair, so that the
        // warps walk 32 pairs at a time whatever the class sizes
        for (int c = warp; c < K; c += kStepThreads / 32) {
            uint32_t s = 0, bits = 0, depth = 0;
            if (lane < nr) {
                const uint4 row = s_rows[lane];
                bits = row.y;
                depth = row.z;
                if (row.w & 1u) {
                    const uint32_t e = tab.get(row.x, (uint32_t)c);
                    if constexpr (STACK) {
                        s = pda_apply(e, bits, depth, maxd, ret);
                    } else {
                        s = e;
                    }
                }
                if constexpr (STACK) {
                    s_cfg4[lane * K + c] = make_uint4(s, bits, depth, 0u);
                } else {
                    s_cfg[lane * K + c] = s;
                }
            }
            const uint32_t live = __ballot_sync(0xffffffffu, s != 0);
            const int n_live = __popc(live);
            const int g0 = s_cls[c], nc = s_cls[c + 1] - g0;
            const int ng = (n_live + kWalkChains - 1) / kWalkChains;
            if (nc > 0 && ng > 0) {
                int base = 0;
                if (lane == 0) base = atomicAdd(&s_ctrl[1], nc * ng);
                base = __shfl_sync(0xffffffffu, base, 0);
                // this lane's row is live row number `rank` of the class
                const int rank = __popc(live & ((1u << lane) - 1u));
                const bool mine = (live >> lane) & 1u;
                for (int g = 0; g < ng; ++g) {
                    const uint32_t part = (mine && (rank >> 2) == g) ? ((uint32_t)lane << (5 * (rank & 3))) : 0u;
                    const uint32_t rows = __reduce_or_sync(0xffffffffu, part) |
                                          ((uint32_t)(min(kWalkChains, n_live - kWalkChains * g) - 1) << 20);
                    for (int k = lane; k < nc; k += 32) s_pairs[base + g * nc + k] = (uint32_t)(g0 + k) | (rows << 10);
                }
            }
        }
        const int eos_local = s_ctrl[2];
        if (tid < nr && eos_local >= 0 && (s_rows[tid].w & 2u)) {
            const int ol = (int)(s_info[eos_local] & 1023u);
            atomicOr(&mt[tid * 32 + (ol >> 5)], 1u << (ol & 31));
            if constexpr (NEXT) s_ntile[tid * kWin + ol] = (uint16_t)s_rows[tid].x;
        }
        __syncthreads();

        prefetch(t + 1);
        const int n_pairs = s_ctrl[1];
        // chunks of 32 pairs: round-robin over the warps, or, for a pushdown
        // automaton (the self-loop skip and the long walks inside strings make
        // chunk times vary) with many chunks per warp, to whichever warp
        // claims the next one
        const bool claim = STACK && n_pairs > 4 * kStepThreads;
        auto next_chunk = [&](int p) {
            if (!claim) return p + kStepThreads;
            int c = 0;
            if (lane == 0) c = atomicAdd(&s_ctrl[4], 1);
            return __shfl_sync(0xffffffffu, c, 0) * 32;
        };
        for (int p0 = claim ? next_chunk(0) : warp * 32; p0 < n_pairs; p0 = next_chunk(p0)) {
            const bool active = p0 + lane < n_pairs;
            const uint32_t pr = active ? s_pairs[p0 + lane] : 0u;
            const int slot = (int)(pr & 1023u);
            const uint32_t info = active ? s_info[slot] : 0u;
            const uint8_t* hp = reinterpret_cast<const uint8_t*>(s_head + 2 * slot);
            const int c = hp[0];   // the token's first class
            const int n_rows = active ? (int)(pr >> 30) + 1 : 0;
            const int len = (int)(info >> 16);
            const int ol = (int)(info & 1023u);
            const uint8_t* tl = len > kInlineBytes ? v.tail + __ldg(v.tail_off + (size_t)w * kWin + slot) : v.tail;
            {
                int rr[kWalkChains];
                uint32_t sv[kWalkChains], bv[kWalkChains], dv[kWalkChains];
#pragma unroll
                for (int k = 0; k < kWalkChains; ++k) {
                    rr[k] = -1;
                    sv[k] = bv[k] = dv[k] = 0u;
                    if (k < n_rows) {
                        rr[k] = (int)((pr >> (10 + 5 * k)) & 31u);
                        if constexpr (STACK) {
                            const uint4 cf = s_cfg4[rr[k] * K + c];
                            sv[k] = cf.x;
                            bv[k] = cf.y;
                            dv[k] = cf.z;
                        } else {
                            sv[k] = s_cfg[rr[k] * K + c];
                        }
                    }
                }
                if (active) {
                    // a token whose later classes all keep every chain's state
                    // leaves the chains as they are: no walk
                    bool keep = use_self;
                    if (use_self) {
                        const unsigned long long tc = s_tokcls[slot];
#pragma unroll
                        for (int k = 0; k < kWalkChains; ++k)
                            if (sv[k] && (tc & ~s_self[sv[k]])) keep = false;
                    }
                    if (!keep) walk_chains<STACK, kWalkChains>(tab, ret, maxd, sv, bv, dv, hp, len, tl);
#pragma unroll
                    for (int k = 0; k < kWalkChains; ++k) {
                        if (rr[k] >= 0 && sv[k]) {
                            atomicOr(&mt[rr[k] * 32 + (ol >> 5)], 1u << (ol & 31));
                            if constexpr (NEXT) s_ntile[rr[k] * kWin + ol] = (uint16_t)sv[k];
                        }
                    }
                }
            }
        }
        if constexpr (NEXT) {
            __syncthreads();
            // coalesced write-out in original-id order
            if (mask) {
                for (int i = tid; i < nr * 32; i += kStepThreads) {
                    const int r = i >> 5, word = w * 32 + (i & 31);
                    if (word < v.W) mask[(size_t)(r0 + r) * v.W + word] = mt[i];
                }
            }
        } else {
            if (t > t0) drain(t - 1, &s_ctrl[0]);
            pw = w;
            pr0 = r0;
            pnr = nr;
        }
        if constexpr (NEXT) {
            const int in_win = min(kWin, v.V - w * kWin);
            if (v.V % 4 == 0) {
                const int per_row = in_win / 4;
                for (int i = tid; i < nr * (kWin / 4); i += kStepThreads) {
                    const int r = i / (kWin / 4), k4 = i % (kWin / 4);
                    if (k4 < per_row) {
                        const uint2 h = reinterpret_cast<const uint2*>(s_ntile + r * kWin)[k4];
                        __stcs(reinterpret_cast<int4*>(next + (size_t)(r0 + r) * v.V + (size_t)w * kWin) + k4,
                               make_int4((int)(h.x & 0xFFFFu), (int)(h.x >> 16), (int)(h.y & 0xFFFFu), (int)(h.y >> 16)));
                    }
                }
            } else {
                for (int i = tid; i < nr * kWin; i += kStepThreads) {
                    const int r = i / kWin, k = i % kWin;
                    if (k < in_win) next[(size_t)(r0 + r) * v.V + (size_t)w * kWin + k] = (int32_t)s_ntile[i];
                }
            }
        }
    }
    if constexpr (!NEXT) {
        if (t1 > t0) {
            __syncthreads();   // the last tile's walk is done
            drain(t1 - 1, &s_ctrl[3]);
        }
    }
}

// ---------------------------------------------------------------------------
// masked argmax / log-sum-exp
// ---------------------------------------------------------------------------
template <bool BF16>
__device__ __forceinline__ float logit_at(const void* row, int t) {
    if constexpr (BF16) {
        const unsigned short u = __ldg(reinterpret_cast<const unsigned short*>(row) + t);
        return __uint_as_float((uint32_t)u << 16);
    } else {
        return __ldg(reinterpret_cast<const float*>(row) + t);
    }
}


// cp.async: 16 bytes global -> shared without a register round trip
__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gmem_src) {
    const unsigned dst = (unsigned)__cvta_generic_to_shared(smem_dst);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(gmem_src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

constexpr int kReduceThreads = 32;            // one warp per CTA: no block barriers

// ---- sampling: Gumbel-max over the allowed logits --------------------------
// Philox4x32-10 (Salmon, Moraes, Dror and Shaw, SC'11): ten rounds of two
// 32x32 -> 64-bit products on the counter, the key advanced by the Weyl
// constants between rounds.
__device__ __forceinline__ uint4 philox10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
    for (int i = 0; i < 10; ++i) {
        const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
        const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
        c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    return c;
}

// ln(x) for a positive normal float: x = 2^e m, m in [sqrt(1/2), sqrt(2)),
// ln x = e ln 2 + 2 atanh(z), z = (m - 1) / (m + 1), with atanh's odd power
// series up to z^11.  Every operation is an explicitly rounded fp32 intrinsic
// (no contraction), so the value is reproducible bit for bit.
__device__ __forceinline__ float ln_rn(float x) {
    const uint32_t bits = __float_as_uint(x);
    int e = (int)((bits >> 23) & 0xFFu) - 127;
    float m = __uint_as_float((bits & 0x7FFFFFu) | 0x3F800000u);
    if (m > 0x1.6a09e6p+0f) {
        m = __fmul_rn(m, 0.5f);
        e += 1;
    }
    const float z = __fdiv_rn(__fsub_rn(m, 1.0f), __fadd_rn(m, 1.0f));
    const float z2 = __fmul_rn(z, z);
    float p = 0x1.745d18p-4f;
    p = __fmaf_rn(p, z2, 0x1.c71c72p-4f);
    p = __fmaf_rn(p, z2, 0x1.24924ap-3f);
    p = __fmaf_rn(p, z2, 0x1.99999ap-3f);
    p = __fmaf_rn(p, z2, 0x1.555556p-2f);
    p = __fmaf_rn(p, z2, 1.0f);
    const float r = __fmul_rn(__fadd_rn(z, z), p);
    const float ef = __int2float_rn(e);
    return __fmaf_rn(ef, 0x1.62e43p-1f, __fmaf_rn(ef, -0x1.05c61p-29f, r));
}

// Gumbel variate of token t of row r: g_t = -ln(-ln(u_t)), u_t = (2k + 1) / 2^24,
// k = (word t % 4 of Philox on (t / 4, r, offset)) >> 9.  `blk` / `rnd` cache
// the last Philox block.
__device__ __forceinline__ float gumbel(const SampleArgs& a, int r, int t, int& blk, uint4& rnd) {
    if ((t >> 2) != blk) {
        blk = t >> 2;
        rnd = philox10(make_uint4((uint32_t)blk, (uint32_t)r, a.off0, a.off1), a.key0, a.key1);
    }
    const uint32_t w = (t & 2) ? ((t & 1) ? rnd.w : rnd.z) : ((t & 1) ? rnd.y : rnd.x);
    const float u = __fmul_rn(__uint2float_rn(2u * (w >> 9) + 1u), 0x1p-24f);
    return -ln_rn(-ln_rn(u));
}

// Every g_t is below this: u_t <= 1 - 2^-24 gives -ln(u_t) >= 5.96e-8 and
// g_t <= 16.64.  A token with x / T + kGumbelMax below the best score so far
// cannot win (rounding is monotonic), so its variate is never drawn.
constexpr float kGumbelMax = 17.0f;

// Where row r's mask words are: row r of `base` ([batch][W]), or, for the
// table-driven step, row states[r] of a precomputed [Q][W] state table.  An
// out-of-range state reads as an all-zero row (nothing allowed) and sets the
// error word.
struct MaskRows {
    const uint32_t* base;       // nullptr (and no row_state): every token allowed
    const int32_t* row_state;   // nullptr: base is [batch][W]
    int32_t Q;
    uint32_t* err;
    __device__ __forceinline__ bool all() const { return base == nullptr; }
    __device__ __forceinline__ const uint32_t* row(int r, int W, bool report) const {
        if (all()) return nullptr;
        if (!row_state) return base + (size_t)r * W;
        const int32_t q = __ldg(row_state + r);
        if (q < 0 || q >= Q) {
            if (report) atomicOr(err, DOMINO_DEVERR_BAD_STATE);
            return nullptr;
        }
        return base + (size_t)q * W;
    }
    // word j of a row given by row(); all-allowed rows read as all ones
    __device__ __forceinline__ uint32_t word(const uint32_t* mrow, int j) const {
        return all() ? 0xFFFFFFFFu : (mrow ? __ldg(mrow + j) : 0u);
    }
};

constexpr int kStageDepth = 3;                // 32-word batches in flight per warp

// Units are mask words (32 tokens); row r holds W units.  Each CTA takes a
// contiguous range of the batch x W units; the CTAs sharing a row leave
// (max, argmax, sum) partials and the last one to finish combines them.
// STAGE (bf16 rows on 16-byte boundaries): a warp takes 32 consecutive words
// of its row at a time; the 16-byte logit vectors that hold an allowed token
// are copied, fully coalesced, into the warp's three-deep staging area
// with cp.async (masks are read four batches ahead, logits two), and each lane
// then folds its own word's allowed logits.  Otherwise each allowed logit is
// read on its own.
// What a row's allowed logits are folded into.
enum Fold : int {
    kFoldLse = 0,      // max, lowest-index argmax and sum of exp (log-sum-exp)
    kFoldMax = 1,      // max and lowest-index argmax only (no lse requested)
    kFoldSample = 2,   // Gumbel-max draw
};

template <bool BF16, bool STAGE, int FOLD>
__global__ void __launch_bounds__(kReduceThreads)
    logits_reduce_kernel(const void* __restrict__ logits, int64_t stride, const MaskRows mask, int V,
                         int W, int B, long long per_cta, float4* __restrict__ partials,
                         uint32_t* __restrict__ counters, int32_t* __restrict__ argmax, float* __restrict__ lse,
                         const SampleArgs sa, int row0, const RowList list) {
    // [buffer][word][16-byte vector]
    __shared__ __align__(16) uint4 stage[STAGE ? kStageDepth * 32 * 4 : 1];
    pdl_wait();
    pdl_trigger();
    const long long N = (long long)list.rows(B) * W;
    const int lane = threadIdx.x;
    long long u = (long long)blockIdx.x * per_cta;
    const long long u_end = min(N, u + per_cta);
    while (u < u_end) {
        const int r = (int)(u / W);
        const long long row_end = (long long)(r + 1) * W;
        const long long seg_end = min(u_end, row_end);
        const int j0 = (int)(u - (long long)r * W), j1 = (int)(seg_end - (long long)r * W);
        const uint32_t* mrow = mask.row(r, W, lane == 0 && j0 == 0);
        const int orow = list.row(r);   // the batch row: logits, outputs and the sampling counter
        const char* lrow = reinterpret_cast<const char*>(logits) + (size_t)orow * stride * (BF16 ? 2 : 4);
        float m = -INFINITY, mL = -INFINITY, s = 0.0f;
        int idx = INT_MAX;
        int blk = -1;                       // Philox block cached by gumbel_score
        uint4 rnd = make_uint4(0u, 0u, 0u, 0u);
        // one allowed logit x of token t (t increasing within a lane)
        auto fold = [&](float x, int t) {
            if constexpr (FOLD == kFoldSample) {
                const float sx = __fmul_rn(x, sa.inv_t);
                if (__fadd_rn(sx, kGumbelMax) < m) return;
                const float sc = __fadd_rn(sx, gumbel(sa, row0 + orow, t, blk, rnd));
                if (sc > m) {
                    m = sc;
                    idx = t;
                }
            } else if constexpr (FOLD == kFoldMax) {
                if (x > m) {
                    m = x;
                    idx = t;
                }
            } else {
                acc_add(m, mL, idx, s, x, t);
            }
        };
        if constexpr (STAGE) {
            const int nb = (j1 - j0 + 31) / 32;   // batches of 32 words
            const int full_words = V / 32;       // words whose 64 bytes of logits lie inside the row
            auto mask_of = [&](int b) -> uint32_t {
                const int j = j0 + 32 * b + lane;
                return (b < nb && j < j1) ? mask.word(mrow, j) : 0u;
            };
            auto issue = [&](int b, uint32_t mw) {
                if (b < nb) {
                    const char* base = lrow + (size_t)(j0 + 32 * b) * 64;
                    uint4* dst = stage + (b % kStageDepth) * 128;
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const int q = 32 * k + lane, wi = q >> 2, sub = q & 3;
                        const uint32_t mq = __shfl_sync(0xffffffffu, mw, wi);
                        if (((mq >> (8 * sub)) & 0xFFu) && j0 + 32 * b + wi < full_words)
                            cp_async16(dst + q, base + (size_t)q * 16);
                    }
                }
                cp_async_commit();
            };
            uint32_t mw[kStageDepth + 1];
#pragma unroll
            for (int k = 0; k <= kStageDepth; ++k) mw[k] = mask_of(k);
#pragma unroll
            for (int k = 0; k < kStageDepth - 1; ++k) issue(k, mw[k]);
            for (int b = 0; b < nb; ++b) {
                issue(b + kStageDepth - 1, mw[kStageDepth - 1]);
                const uint32_t mw_far = mask_of(b + kStageDepth + 1);
                cp_async_wait<kStageDepth - 1>();   // batch b has landed
                __syncwarp();
                const int j = j0 + 32 * b + lane;
                uint32_t word = mw[0];
                if (word) {
                    const int t0 = j * 32;
                    if (FOLD != kFoldSample && j < full_words && __popc(word) > 12) {
                        // a dense word: the word's maximum first (every token compared in
                        // order, no bit scan), then, for the log-sum-exp, one rescale and
                        // the sum of the word's terms
                        const uint4* sv = stage + (b % kStageDepth) * 128 + lane * 4;
                        uint32_t qs[16];
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const uint4 q = ((word >> (8 * k)) & 0xFFu) ? sv[k] : make_uint4(0u, 0u, 0u, 0u);
                            qs[4 * k] = q.x;
                            qs[4 * k + 1] = q.y;
                            qs[4 * k + 2] = q.z;
                            qs[4 * k + 3] = q.w;
                        }
                        float wm = -INFINITY;
                        int wi = 0;
#pragma unroll
                        for (int e = 0; e < 32; ++e) {
                            const float x = (e & 1) ? bf16_hi(qs[e >> 1]) : bf16_lo(qs[e >> 1]);
                            if (((word >> e) & 1u) && x > wm) {
                                wm = x;
                                wi = e;
                            }
                        }
                        if constexpr (FOLD == kFoldMax) {
                            if (wm > m) {
                                m = wm;
                                idx = t0 + wi;
                            }
                        } else {
                            if (wm > m) {   // earlier words hold lower ids: equal maxima keep idx
                                const float wL = wm * kLog2e;
                                s = s == 0.0f ? 0.0f : s * ex2(mL - wL);
                                m = wm;
                                mL = wL;
                                idx = t0 + wi;
                            }
                            float acc = 0.0f;
#pragma unroll
                            for (int e = 0; e < 32; ++e) {
                                const float x = (e & 1) ? bf16_hi(qs[e >> 1]) : bf16_lo(qs[e >> 1]);
                                acc += ((word >> e) & 1u) ? ex2(fmaf(x, kLog2e, -mL)) : 0.0f;
                            }
                            s += acc;
                        }
                    } else if (j < full_words) {
                        const unsigned short* st =
                            reinterpret_cast<const unsigned short*>(stage + (b % kStageDepth) * 128 + lane * 4);
                        while (word) {
                            const int e = __ffs(word) - 1;
                            word &= word - 1;
                            fold(__uint_as_float((uint32_t)st[e] << 16), t0 + e);
                        }
                    } else {   // the row's partial last word
                        while (word) {
                            const int e = __ffs(word) - 1;
                            word &= word - 1;
                            if (t0 + e < V) fold(logit_at<BF16>(lrow, t0 + e), t0 + e);
                        }
                    }
                }
                __syncwarp();   // this buffer is refilled by the next issue
#pragma unroll
                for (int k = 0; k < kStageDepth; ++k) mw[k] = mw[k + 1];
                mw[kStageDepth] = mw_far;
            }
            cp_async_wait<0>();
        } else {
            for (int j = j0 + lane; j < j1; j += 32) {
                uint32_t word = mask.word(mrow, j);
                const int t0 = j * 32;
                while (word) {
                    const int e = __ffs(word) - 1;
                    word &= word - 1;
                    if (t0 + e < V) fold(logit_at<BF16>(lrow, t0 + e), t0 + e);
                }
            }
        }
        warp_merge(m, idx, s);
        const long long first = ((long long)r * W) / per_cta;
        const long long last = (row_end - 1) / per_cta;
        const int nseg = (int)(last - first + 1);
        bool is_last = false;
        if (lane == 0) {
            if (nseg == 1) {
                argmax[orow] = m == -INFINITY ? -1 : idx;
                if (lse) lse[orow] = m == -INFINITY ? -INFINITY : m + logf(s);
            } else {
                partials[(size_t)r * kMaxSegments + (blockIdx.x - first)] =
                    make_float4(m, __int_as_float(idx), s, 0.f);
                __threadfence();
                is_last = atomicAdd(counters + r, 1u) == (unsigned)(nseg - 1);
            }
        }
        if (__shfl_sync(0xffffffffu, is_last, 0)) {
            // last CTA of the row: combine its segments
            __threadfence();
            m = -INFINITY;
            s = 0.0f;
            idx = INT_MAX;
            for (int k = lane; k < nseg; k += 32) {
                const float4 p = __ldcg(partials + (size_t)r * kMaxSegments + k);
                acc_merge(m, idx, s, p.x, __float_as_int(p.y), p.z);
            }
            warp_merge(m, idx, s);
            if (lane == 0) {
                argmax[orow] = m == -INFINITY ? -1 : idx;
                if (lse) lse[orow] = m == -INFINITY ? -INFINITY : m + logf(s);
                counters[r] = 0u;   // ready for the next launch (stream-ordered)
            }
        }
        u = seg_end;
    }
}

// ---- the greedy / log-sum-exp pass over bf16 rows: a compacted gather -----
// One CTA per row, its warps (up to 16) on consecutive segments of the row's
// mask words, each segment cut into spans of 32 x kGatherSpan words (lane l
// holds words l*kGatherSpan ... +kGatherSpan-1 of the span).  Each lane finds
// its words' 16-byte logit vectors that hold an allowed token (a 32-bit map,
// one bit per vector), a warp scan places the lanes' lists one after the
// other in token order, and the warp then loads the listed vectors
// kGatherRound per lane at once (entry k goes to lane k % 32, so each lane
// still sees its tokens in increasing order) and folds them.  Zero words cost
// a few instructions, every load of a span is independent, and a span costs
// one memory latency whatever its density.  The warps' partials are merged in
// shared memory.  Logit lines are not kept in L1, and in L2 only when a
// log-prob pass reads them again (evict-last; otherwise evict-first).
constexpr int kGatherMaxWarps = 16;   // warps per CTA (one row); two CTAs per SM
constexpr int kGatherSpan = 8;     // mask words per lane per span (8192 tokens)
constexpr int kGatherWarpSmem = 32 * kGatherSpan * (4 + 4 * 2);   // a span's words and its list
constexpr int kGatherRound = 4;    // vectors per lane loaded together

__device__ __forceinline__ uint64_t l2_policy(bool keep) {
    uint64_t p;
    if (keep)
        asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;\n" : "=l"(p));
    else
        asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;\n" : "=l"(p));
    return p;
}

__device__ __forceinline__ uint4 ld_once16(const void* p, uint64_t pol) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;\n"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p), "l"(pol));
    return v;
}

// bit b of the result: byte b of x is not zero
__device__ __forceinline__ uint32_t nonzero_bytes(uint32_t x) {
    x |= x >> 4;
    x |= x >> 2;
    x |= x >> 1;
    return ((x & 0x01010101u) * 0x10204080u) >> 28;
}

// element e (0..7) of eight bf16 values
__device__ __forceinline__ float bf16_of(const uint4& q, int e) {
    const uint32_t h = (e & 4) ? ((e & 2) ? q.w : q.z) : ((e & 2) ? q.y : q.x);
    return (e & 1) ? bf16_hi(h) : bf16_lo(h);
}

// chunk: words per warp, a multiple of kGatherSpan.  A sampling pass draws
// row r with counter row row0 + (batch row of r).
template <int FOLD>
__global__ void __launch_bounds__(kGatherMaxWarps * 32, 2)
    logits_gather_kernel(const void* __restrict__ logits, int64_t stride, const MaskRows mask, int V, int W, int B,
                         int chunk, int32_t* __restrict__ argmax, float* __restrict__ lse, const SampleArgs sa,
                         int row0, int keep_l2, const RowList list) {
    constexpr int kSpanWords = 32 * kGatherSpan;
    extern __shared__ __align__(16) unsigned char g_smem[];   // per warp: words, then list
    __shared__ float4 s_part[kGatherMaxWarps];
    pdl_wait();
    pdl_trigger();
    const int r = blockIdx.x;
    if (r >= list.rows(B)) return;   // the whole CTA
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    uint32_t* sw = reinterpret_cast<uint32_t*>(g_smem + wid * kGatherWarpSmem);   // a span's mask words
    uint16_t* lst = reinterpret_cast<uint16_t*>(sw + kSpanWords);                // its vectors, in token order
    const uint64_t pol = l2_policy(keep_l2 != 0);
    const int full_vec = V / 8;   // vectors that lie wholly inside the row
    const int j0 = wid * chunk, j1 = min(W, j0 + chunk);
    const uint32_t* mrow = mask.row(r, W, threadIdx.x == 0);
    const int orow = list.row(r);
    const char* lrow = reinterpret_cast<const char*>(logits) + (size_t)orow * stride * 2;
    float m = -INFINITY, mL = -INFINITY, s = 0.0f;
    int idx = INT_MAX;
    int blk = -1;   // Philox block cached by gumbel()
    uint4 rnd = make_uint4(0u, 0u, 0u, 0u);
    // one allowed logit x of token t (t increasing within a lane)
    auto fold1 = [&](float x, int t) {
        if constexpr (FOLD == kFoldSample) {
            const float sx = __fmul_rn(x, sa.inv_t);
            if (__fadd_rn(sx, kGumbelMax) < m) return;
            const float sc = __fadd_rn(sx, gumbel(sa, row0 + orow, t, blk, rnd));
            if (sc > m) {
                m = sc;
                idx = t;
            }
        } else if constexpr (FOLD == kFoldMax) {
            if (x > m) {
                m = x;
                idx = t;
            }
        } else {
            acc_add(m, mL, idx, s, x, t);
        }
    };
    for (int js = j0; js < j1; js += kSpanWords) {
        uint32_t w[kGatherSpan];
        const int jl = js + lane * kGatherSpan;
        if (mrow && jl + kGatherSpan <= j1 && (reinterpret_cast<uintptr_t>(mrow + jl) & 15) == 0) {
            const uint4 a = __ldg(reinterpret_cast<const uint4*>(mrow + jl));
            const uint4 b = __ldg(reinterpret_cast<const uint4*>(mrow + jl) + 1);
            w[0] = a.x, w[1] = a.y, w[2] = a.z, w[3] = a.w, w[4] = b.x, w[5] = b.y, w[6] = b.z, w[7] = b.w;
        } else {
#pragma unroll
            for (int g = 0; g < kGatherSpan; ++g) w[g] = jl + g < j1 ? mask.word(mrow, jl + g) : 0u;
        }
        uint32_t nb = 0;   // bit 4g + b: byte b of word g holds an allowed token
#pragma unroll
        for (int g = 0; g < kGatherSpan; ++g) nb |= nonzero_bytes(w[g]) << (4 * g);
        reinterpret_cast<uint4*>(sw)[2 * lane] = make_uint4(w[0], w[1], w[2], w[3]);
        reinterpret_cast<uint4*>(sw)[2 * lane + 1] = make_uint4(w[4], w[5], w[6], w[7]);
        const int c = __popc(nb);
        int incl = c;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off) incl += y;
        }
        const int T = __shfl_sync(0xffffffffu, incl, 31);
        if (T == 0) continue;   // warp-uniform
        int pos = incl - c;
        while (nb) {
            const int bit = __ffs(nb) - 1;
            nb &= nb - 1;
            lst[pos++] = (uint16_t)(lane * 4 * kGatherSpan + bit);
        }
        __syncwarp();
        const int vbase = js * 4;   // the span's first vector in the row
        // rounds of kGatherRound vectors per lane; the next round's loads are
        // issued before this round is folded
        int ent[kGatherRound];
        uint4 q[kGatherRound];
        auto load_round = [&](int k0, int(&en)[kGatherRound], uint4(&qq)[kGatherRound]) {
#pragma unroll
            for (int i = 0; i < kGatherRound; ++i) {
                const int k = k0 + i * 32 + lane;
                en[i] = k < T ? (int)lst[k] : -1;
                const int vi = vbase + en[i];
                qq[i] = (en[i] >= 0 && vi < full_vec) ? ld_once16(lrow + (size_t)vi * 16, pol)
                                                     : make_uint4(0u, 0u, 0u, 0u);
            }
        };
        load_round(0, ent, q);
        for (int k0 = 0; k0 < T; k0 += 32 * kGatherRound) {
            int ent_n[kGatherRound];
            uint4 q_n[kGatherRound];
            const bool more = k0 + 32 * kGatherRound < T;   // warp-uniform
            if (more) load_round(k0 + 32 * kGatherRound, ent_n, q_n);
#pragma unroll
            for (int i = 0; i < kGatherRound; ++i) {
                if (ent[i] < 0) continue;
                const int vi = vbase + ent[i], t0 = vi * 8;
                uint32_t bm = (sw[ent[i] >> 2] >> (8 * (ent[i] & 3))) & 0xFFu;
                if (vi >= full_vec) {   // the row's last, partial vector: token by token
                    while (bm) {
                        const int e = __ffs(bm) - 1;
                        bm &= bm - 1;
                        if (t0 + e >= V) break;
                        fold1(logit_at<true>(lrow, t0 + e), t0 + e);
                    }
                } else if (FOLD == kFoldSample) {
                    while (bm) {
                        const int e = __ffs(bm) - 1;
                        bm &= bm - 1;
                        fold1(bf16_of(q[i], e), t0 + e);
                    }
                } else if (__popc(bm) > 2) {
                    // a dense vector: its allowed maximum (first on ties), one
                    // rescale, then its sum, all eight lanes of it predicated;
                    // earlier vectors hold lower ids, so an equal maximum keeps idx
                    float xs[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) xs[e] = ((bm >> e) & 1u) ? bf16_of(q[i], e) : -INFINITY;
                    float vm = xs[0];
                    int ve = 0;
#pragma unroll
                    for (int e = 1; e < 8; ++e)
                        if (xs[e] > vm) {
                            vm = xs[e];
                            ve = e;
                        }
                    if constexpr (FOLD == kFoldMax) {
                        if (vm > m) {
                            m = vm;
                            idx = t0 + ve;
                        }
                    } else {
                        if (vm > m) {
                            const float vL = vm * kLog2e;
                            s = s == 0.0f ? 0.0f : s * ex2(mL - vL);
                            m = vm;
                            mL = vL;
                            idx = t0 + ve;
                        }
                        float acc = 0.0f;
#pragma unroll
                        for (int e = 0; e < 8; ++e) acc += ((bm >> e) & 1u) ? ex2(fmaf(xs[e], kLog2e, -mL)) : 0.0f;
                        s += acc;
                    }
                } else {
                    while (bm) {
                        const int e = __ffs(bm) - 1;
                        bm &= bm - 1;
                        fold1(bf16_of(q[i], e), t0 + e);
                    }
                }
            }
            if (more) {
#pragma unroll
                for (int i = 0; i < kGatherRound; ++i) {
                    ent[i] = ent_n[i];
                    q[i] = q_n[i];
                }
            }
        }
        __syncwarp();   // the span buffers are rewritten by the next span
    }
    warp_merge(m, idx, s);
    if (lane == 0) s_part[wid] = make_float4(m, __int_as_float(idx), s, 0.f);
    __syncthreads();
    if (wid == 0) {
        m = -INFINITY;
        s = 0.0f;
        idx = INT_MAX;
        if (lane < nwarps) {
            const float4 p = s_part[lane];
            m = p.x;
            idx = __float_as_int(p.y);
            s = p.z;
        }
        warp_merge(m, idx, s);
        if (lane == 0) {
            argmax[orow] = m == -INFINITY ? -1 : idx;
            if (lse) lse[orow] = m == -INFINITY ? -INFINITY : m + logf(s);
        }
    }
}

// logprob[t] = logit[t] - lse for allowed t, -inf otherwise.  VEC (bf16 rows on
// 16-byte boundaries, V % 4 == 0): a thread takes 16 consecutive tokens when
// V % 16 == 0 (32 bytes of logits read unconditionally, four float4 stores),
// else 4 (their 8 bytes read only when one is allowed, one float4 store);
// grid-stride over the batch's groups.  Otherwise one mask word (32 tokens) per
// thread, one token at a time.
template <bool BF16, bool VEC>
__global__ void __launch_bounds__(kLogitThreads)
    logprobs_kernel(const void* __restrict__ logits, int64_t stride, const MaskRows mask, int V, int W,
                    int B, const float* __restrict__ lse, float* __restrict__ out, int wide) {
    pdl_wait();
    pdl_trigger();
    if (VEC && BF16 && V % 16 == 0) {
        // 16 tokens per thread: two 16-byte logit loads and the mask half-word,
        // all independent, then four float4 stores
        const int ng = V / 16;
        const long long N = (long long)B * ng;
        for (long long u = (long long)blockIdx.x * kLogitThreads + threadIdx.x; u < N;
             u += (long long)gridDim.x * kLogitThreads) {
            const int r = (int)(u / ng), g = (int)(u - (long long)r * ng);
            const uint32_t* mrow = mask.row(r, W, false);
            const char* lrow = reinterpret_cast<const char*>(logits) + (size_t)r * stride * 2;
            const uint4* src = reinterpret_cast<const uint4*>(lrow) + 2 * (size_t)g;
            uint32_t ws[8];
            if (wide) {   // one 32-byte load (32-byte aligned rows)
                asm volatile("ld.global.cs.v8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                             : "=r"(ws[0]), "=r"(ws[1]), "=r"(ws[2]), "=r"(ws[3]), "=r"(ws[4]), "=r"(ws[5]),
                               "=r"(ws[6]), "=r"(ws[7])
                             : "l"(src));
            } else {
                const uint4 a = __ldcs(src), c = __ldcs(src + 1);
                ws[0] = a.x; ws[1] = a.y; ws[2] = a.z; ws[3] = a.w;
                ws[4] = c.x; ws[5] = c.y; ws[6] = c.z; ws[7] = c.w;
            }
            const uint32_t bits = (mask.word(mrow, g >> 1) >> (16 * (g & 1))) & 0xFFFFu;
            const float l = __ldg(lse + r);
            float o[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const float x = (e & 1) ? bf16_hi(ws[e >> 1]) : bf16_lo(ws[e >> 1]);
                o[e] = ((bits >> e) & 1u) ? x - l : -INFINITY;
            }
            float* dst = out + (size_t)r * V + 16 * (size_t)g;
            if (wide) {   // two 32-byte stores
#pragma unroll
                for (int h = 0; h < 2; ++h)
                    asm volatile("st.global.cs.v8.f32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"l"(dst + 8 * h),
                                 "f"(o[8 * h]), "f"(o[8 * h + 1]), "f"(o[8 * h + 2]), "f"(o[8 * h + 3]),
                                 "f"(o[8 * h + 4]), "f"(o[8 * h + 5]), "f"(o[8 * h + 6]), "f"(o[8 * h + 7])
                                 : "memory");
            } else {
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    __stcs(reinterpret_cast<float4*>(dst) + q, make_float4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]));
            }
        }
    } else if constexpr (VEC && BF16) {
        const int nq = V / 4;
        const long long N = (long long)B * nq;
        for (long long u = (long long)blockIdx.x * kLogitThreads + threadIdx.x; u < N;
             u += (long long)gridDim.x * kLogitThreads) {
            const int r = (int)(u / nq), qd = (int)(u - (long long)r * nq);
            const uint32_t* mrow = mask.row(r, W, false);
            const uint32_t nib = (mask.word(mrow, qd >> 3) >> (4 * (qd & 7))) & 0xFu;
            float4 o = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
            if (nib) {
                const char* lrow = reinterpret_cast<const char*>(logits) + (size_t)r * stride * 2;
                const uint2 v = __ldcs(reinterpret_cast<const uint2*>(lrow) + qd);
                const float l = __ldg(lse + r);
                if (nib & 1u) o.x = bf16_lo(v.x) - l;
                if (nib & 2u) o.y = bf16_hi(v.x) - l;
                if (nib & 4u) o.z = bf16_lo(v.y) - l;
                if (nib & 8u) o.w = bf16_hi(v.y) - l;
            }
            __stcs(reinterpret_cast<float4*>(out + (size_t)r * V) + qd, o);
        }
    } else {
        const long long N = (long long)B * W;
        for (long long u = (long long)blockIdx.x * kLogitThreads + threadIdx.x; u < N;
             u += (long long)gridDim.x * kLogitThreads) {
            const int r = (int)(u / W), j = (int)(u - (long long)r * W);
            const uint32_t* mrow = mask.row(r, W, false);
            const uint32_t word = mask.word(mrow, j);
            const char* lrow = reinterpret_cast<const char*>(logits) + (size_t)r * stride * (BF16 ? 2 : 4);
            float* orow = out + (size_t)r * V + (size_t)j * 32;
            const float l = __ldg(lse + r);
            for (int e = 0; e < 32 && j * 32 + e < V; ++e)
                orow[e] = ((word >> e) & 1u) ? logit_at<BF16>(lrow, j * 32 + e) - l : -INFINITY;
        }
    }
}

// ---------------------------------------------------------------------------
// advance
// ---------------------------------------------------------------------------
template <bool STACK, int MODE>
__global__ void __launch_bounds__(kAdvanceThreads)
    advance_kernel(const StepView v, const uint4* __restrict__ img, int img_words, int tgt_off, int ret_off,
                   const int32_t* states, const uint64_t* stacks, const int32_t* __restrict__ tokens, int32_t batch,
                   int32_t* states_out, uint64_t* stacks_out) {
    using E = typename std::conditional<STACK, uint32_t, uint16_t>::type;
    extern __shared__ __align__(16) unsigned char adv_smem[];
    if constexpr (MODE != kDenseGlobal) {
        // the table image (written at load time, by no kernel) is staged
        // before the launch wait, while the kernel before this one drains
        for (int i = threadIdx.x; i < img_words; i += kAdvanceThreads)
            reinterpret_cast<uint4*>(adv_smem)[i] = __ldg(img + i);
        __syncthreads();
    }
    pdl_wait();
    pdl_trigger();
    const int b = blockIdx.x * kAdvanceThreads + threadIdx.x;
    if (b >= batch) return;
    if constexpr (MODE == kDenseGlobal) {
        advance_row<STACK, kDenseGlobal>(v, states, stacks, b, tokens[b], states_out, stacks_out);
    } else {
        Tab<E, MODE> tab;
        tab.dense = reinterpret_cast<const E*>(adv_smem);
        tab.sp = reinterpret_cast<const uint32_t*>(adv_smem);
        tab.tgt = reinterpret_cast<const E*>(adv_smem + tgt_off);
        tab.K = (uint32_t)v.K;
        debug_bounds(tab, v);
        advance_row_with<STACK>(v, tab, reinterpret_cast<const uint16_t*>(adv_smem + ret_off), states, stacks, b,
                                tokens[b], states_out, stacks_out);
    }
}

// Opportunistic masking, the check: is row b's proposal (its unmasked argmax)
// allowed from the row's configuration?  The same rule as the mask: the walk
// stays live; EOS needs an accepting state and an empty stack; other empty
// tokens never pass.  Allowed proposals are the row's decoded token; rejected
// (and invalid) rows are appended to the fallback list.
template <bool STACK, int MODE>
__global__ void __launch_bounds__(kAdvanceThreads)
    propose_check_kernel(const StepView v, const int32_t* __restrict__ states, const uint64_t* __restrict__ stacks,
                         const int32_t* __restrict__ proposals, int32_t batch, int32_t* __restrict__ tokens_out,
                         int32_t* __restrict__ row_ids, int32_t* __restrict__ row_count) {
    using E = typename std::conditional<STACK, uint32_t, uint16_t>::type;
    pdl_wait();
    pdl_trigger();
    const int b = blockIdx.x * kAdvanceThreads + threadIdx.x;
    if (b >= batch) return;
    const int32_t t = proposals[b];
    bool ok = false;
    if (t >= 0 && t < v.V) {
        const uint4 rc = read_row(v, states, stacks, b, false);   // the fallback reports invalid rows
        if (rc.w & 1u) {
            if (t == v.eos_id) {
                ok = (rc.w & 2u) != 0u;
            } else {
                Tab<E, MODE == kDenseSmem ? kDenseGlobal : MODE> tab;
                tab.dense = reinterpret_cast<const E*>(STACK ? (const void*)v.t32 : (const void*)v.t16);
                tab.sp = v.sp_info;
                tab.tgt = reinterpret_cast<const E*>(v.sp_tgt);
                tab.K = (uint32_t)v.K;
                debug_bounds(tab, v);
                const int p = __ldg(v.pos_of + t);
                const int len = (int)(__ldg(v.info + p) >> 16);
                if (len > 0) {
                    const uint8_t* hp = reinterpret_cast<const uint8_t*>(v.head + 2 * (size_t)p);
                    const uint8_t* tail = len > kInlineBytes ? v.tail + __ldg(v.tail_off + p) : v.tail;
                    uint32_t bits = rc.y, depth = rc.z;
                    ok = walk<STACK, 0>(tab, v.ret, (uint32_t)v.max_depth, rc.x, bits, depth, hp, len, tail) != 0u;
                }
            }
        }
    }
    if (ok) {
        tokens_out[b] = t;
    } else {
        row_ids[atomicAdd(row_count, 1)] = b;
    }
}

// ---- count-based speculation (Sec. 3.6) ------------------------------------
// The count model is keyed by (scanner state, top of the bracket stack):
// key = state for a DFA, state * 3 + top for a pushdown automaton (top 0: empty
// stack, 1 + symbol otherwise).  best[key] packs the largest count with the
// complement of its token id, so atomicMax keeps the most frequent token and,
// on equal counts, the lowest id, whatever order the updates come in.
__device__ __forceinline__ uint32_t spec_key(bool stack, uint32_t s, uint32_t bits, uint32_t depth) {
    if (!stack) return s;
    return s * 3u + (depth == 0 ? 0u : 1u + (bits & 1u));
}

template <bool STACK>
__global__ void __launch_bounds__(kAdvanceThreads)
    spec_update_kernel(const StepView v, const int32_t* __restrict__ states, const uint64_t* __restrict__ stacks,
                       const int32_t* __restrict__ tokens, int32_t batch, uint32_t* __restrict__ counts,
                       unsigned long long* __restrict__ best, uint32_t* __restrict__ reached) {
    pdl_wait();
    pdl_trigger();
    const int b = blockIdx.x * kAdvanceThreads + threadIdx.x;
    if (b >= batch) return;
    const int32_t t = tokens[b];
    if (t < 0 || t >= v.V) return;
    const uint4 rc = read_row(v, states, stacks, b, false);
    if (!(rc.w & 1u)) return;
    const uint32_t key = spec_key(STACK, rc.x, rc.y, rc.z);
    atomicAdd(reached + key, 1u);
    const uint32_t c = atomicAdd(counts + (size_t)key * v.V + t, 1u) + 1u;
    atomicMax(best + key, ((unsigned long long)c << 32) | (0xFFFFFFFFu - (uint32_t)t));
}

// Up to s proposals per row, each the key's most frequent token while
// count * 1000 >= min_permille * reached; a proposal must be allowed from the
// chain's configuration (walked; EOS needs an accepting state and an empty
// stack, and ends the chain).  chain_* [batch][s + 1]: configurations after
// 0..s proposals, the last one repeated past the chain's end.
template <bool STACK, int MODE>
__global__ void __launch_bounds__(kAdvanceThreads)
    spec_propose_kernel(const StepView v, const int32_t* __restrict__ states, const uint64_t* __restrict__ stacks,
                        int32_t batch, int32_t s, int32_t min_permille, const unsigned long long* __restrict__ best,
                        const uint32_t* __restrict__ reached, int32_t* __restrict__ proposals,
                        int32_t* __restrict__ n_prop, int32_t* __restrict__ chain_states,
                        uint64_t* __restrict__ chain_stacks) {
    using E = typename std::conditional<STACK, uint32_t, uint16_t>::type;
    pdl_wait();
    pdl_trigger();
    const int b = blockIdx.x * kAdvanceThreads + threadIdx.x;
    if (b >= batch) return;
    Tab<E, MODE == kDenseSmem ? kDenseGlobal : MODE> tab;
    tab.dense = reinterpret_cast<const E*>(STACK ? (const void*)v.t32 : (const void*)v.t16);
    tab.sp = v.sp_info;
    tab.tgt = reinterpret_cast<const E*>(v.sp_tgt);
    tab.K = (uint32_t)v.K;
    debug_bounds(tab, v);
    const int32_t sv = __ldg(states + b);
    const unsigned long long wv = stacks ? __ldg(reinterpret_cast<const unsigned long long*>(stacks) + b) : 0ull;
    const uint4 rc = decode_row(v, sv, wv, stacks != nullptr, v.accept_bits, false);
    uint32_t q = rc.x, bits = rc.y, depth = rc.z;
    int n = 0;
    int32_t* prow = proposals + (size_t)b * s;
    int32_t* crow = chain_states + (size_t)b * (s + 1);
    uint64_t* krow = chain_stacks ? chain_stacks + (size_t)b * (s + 1) : nullptr;
    crow[0] = sv;
    if (krow) krow[0] = wv;
    bool go = (rc.w & 1u) != 0u;
    while (go && n < s) {
        const uint32_t key = spec_key(STACK, q, bits, depth);
        const uint32_t R = __ldg(reached + key);
        const unsigned long long bk = __ldg(best + key);
        const uint32_t c = (uint32_t)(bk >> 32);
        const int32_t t = (int32_t)(0xFFFFFFFFu - (uint32_t)bk);
        if (R == 0u || c == 0u || (unsigned long long)c * 1000ull < (unsigned long long)min_permille * R) break;
        if (t == v.eos_id) {
            const bool acc = depth == 0 && ((__ldg(v.accept_bits + (q >> 5)) >> (q & 31u)) & 1u);
            if (!acc) break;
            prow[n] = t;
            ++n;
            crow[n] = (int32_t)q;
            if (krow) krow[n] = ((uint64_t)depth << 32) | bits;
            break;
        }
        const int p = __ldg(v.pos_of + t);
        const int len = (int)(__ldg(v.info + p) >> 16);
        if (len == 0) break;
        const uint8_t* hp = reinterpret_cast<const uint8_t*>(v.head + 2 * (size_t)p);
        const uint8_t* tail = len > kInlineBytes ? v.tail + __ldg(v.tail_off + p) : v.tail;
        uint32_t nb = bits, nd = depth;
        const uint32_t nq = walk<STACK, 0>(tab, v.ret, (uint32_t)v.max_depth, q, nb, nd, hp, len, tail);
        if (nq == 0u) break;
        prow[n] = t;
        q = nq;
        bits = nb;
        depth = nd;
        ++n;
        crow[n] = (int32_t)q;
        if (krow) krow[n] = ((uint64_t)depth << 32) | bits;
    }
    n_prop[b] = n;
    for (int i = n; i < s; ++i) prow[i] = -1;
    for (int i = n + 1; i <= s; ++i) {
        crow[i] = crow[n];
        if (krow) krow[i] = krow[n];
    }
}

// n_accept[b]: leading proposals equal to the constrained decode at their
// chain configuration; tokens_out[b] the decode after them and
// states_out / stacks_out the chain configuration it is decoded from.
__global__ void __launch_bounds__(kAdvanceThreads)
    spec_accept_kernel(const int32_t* __restrict__ proposals, const int32_t* __restrict__ n_prop,
                       const int32_t* __restrict__ decoded, const int32_t* __restrict__ chain_states,
                       const uint64_t* __restrict__ chain_stacks, int32_t batch, int32_t s,
                       int32_t* __restrict__ n_accept, int32_t* __restrict__ tokens_out,
                       int32_t* __restrict__ states_out, uint64_t* __restrict__ stacks_out) {
    pdl_wait();
    pdl_trigger();
    const int b = blockIdx.x * kAdvanceThreads + threadIdx.x;
    if (b >= batch) return;
    const int n = n_prop[b];
    int k = 0;
    while (k < n && decoded[(size_t)b * (s + 1) + k] == proposals[(size_t)b * s + k]) ++k;
    n_accept[b] = k;
    if (tokens_out) tokens_out[b] = decoded[(size_t)b * (s + 1) + k];
    if (states_out) states_out[b] = chain_states[(size_t)b * (s + 1) + k];
    if (stacks_out && chain_stacks) stacks_out[b] = chain_stacks[(size_t)b * (s + 1) + k];
}


// Alg. 1 update from the precomputed state x token table: one read of
// next[s][t] per sequence (EOS or -1: the start state; a rejected token's
// entry is 0, the dead state).  states_out may alias states: each thread reads
// its row before writing it.
__global__ void __launch_bounds__(kAdvanceThreads)
    advance_table_kernel(const int32_t* __restrict__ table_next, int32_t Q, int32_t V, int32_t eos_id, int32_t start,
                         const int32_t* states, const int32_t* __restrict__ tokens, int32_t batch,
                         int32_t* states_out, uint32_t* __restrict__ err) {
    pdl_wait();
    pdl_trigger();
    const int b = blockIdx.x * kAdvanceThreads + threadIdx.x;
    if (b >= batch) return;
    const int32_t t = tokens[b];
    int32_t s = 0;
    if (t < 0 || t == eos_id) {
        s = start;
    } else if (t >= V) {
        atomicOr(err, DOMINO_DEVERR_BAD_TOKEN);
    } else {
        const int32_t q = states[b];
        if (q < 0 || q >= Q) atomicOr(err, DOMINO_DEVERR_BAD_STATE);
        else s = __ldg(table_next + (size_t)q * V + t);
    }
    states_out[b] = s;
}

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------
// Rows per tile: as many as possible (<= 32, one ballot) while the tiles
// still split evenly over one CTA per SM.
// With next states, the [R][1024] staging tile of next states decides: as many
// rows as shared memory holds (the table placement was chosen for R = 8).
int rows_per_tile(const StepView& v, const LaunchEnv& env, int batch, bool next, bool stack, int img_bytes) {
    if (next) {
        for (int R = kMaxRowsPerTile; R > kRowsPerTileNext; R >>= 1)
            if (step_layout(v.K, R, true, stack, v.Q, img_bytes, v.self_mask != nullptr).total <=
                    env.max_smem_optin &&
                (long long)((batch + R - 1) / R) * v.n_windows >= 4LL * env.num_sms)
                return R;
        return kRowsPerTileNext;
    }
    int best = kRowsPerTile;
    double best_waste = 1e9;
    for (int R = kMaxRowsPerTile; R >= kRowsPerTile; R -= 4) {
        const long long tiles = (long long)((batch + R - 1) / R) * v.n_windows;
        const double per = (double)tiles / env.num_sms;
        const double waste = tiles < env.num_sms ? 1.0 - per : (double)((tiles + env.num_sms - 1) / env.num_sms) / per - 1.0;
        if (waste < 0.08) return R;
        if (waste < best_waste) {
            best_waste = waste;
            best = R;
        }
    }
    return best;
}

template <bool STACK, int MODE, bool NEXT>
cudaError_t launch_step_t(const StepView& v, const LaunchEnv& env, const int32_t* states, const uint64_t* stacks,
                          int32_t batch, bool row_is_state, uint32_t* mask, int32_t* next, const RowList& list,
                          const FuseArgs& fuse, cudaStream_t st) {
    const int img_bytes = MODE == kDenseGlobal ? 0 : (int)table_smem_bytes(v, STACK, MODE);
    const int R = rows_per_tile(v, env, batch, NEXT, STACK, img_bytes);
    const StepLayout L = step_layout(v.K, R, NEXT, STACK, v.Q, img_bytes, v.self_mask != nullptr);
    auto kern = step_kernel<STACK, MODE, NEXT>;
    // the dynamic shared-memory limit is raised once per device and size, so
    // that launches inside a stream capture make no attribute calls
    static int configured[kMaxDevices] = {0};
    static std::mutex mu;   // handles on different host threads share it
    int dev = 0;
    cudaGetDevice(&dev);
    if (L.total > 48 * 1024 && dev < kMaxDevices) {
        std::lock_guard<std::mutex> lk(mu);
        if (configured[dev] < L.total) {
            cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L.total);
            if (e != cudaSuccess) return e;
            configured[dev] = L.total;
        }
    }
    const int n_row_tiles = (batch + R - 1) / R;
    const int n_tiles = n_row_tiles * v.n_windows;
    const int grid = min(n_tiles, env.num_sms);
    const uint4* img = nullptr;
    int tgt_off = 0, ret_off = 0;
    if constexpr (MODE != kDenseGlobal) {
        const size_t esz = STACK ? 4 : 2;
        if (MODE == kDenseSmem) {
            img = reinterpret_cast<const uint4*>(STACK ? (const void*)v.t32 : (const void*)v.t16);
            ret_off = align16((int)((size_t)v.Q * v.K * esz));
        } else {
            img = reinterpret_cast<const uint4*>(v.sp_info);
            tgt_off = align16(v.Q * (MODE == kSparse32Smem ? 8 : 16));
            ret_off = tgt_off + align16((int)((size_t)v.sp_nnz * esz));
        }
    }
    return launch_pdl(kern, dim3(grid), dim3(kStepThreads), (size_t)L.total, st, v, img, img_bytes, tgt_off, ret_off,
                      states, stacks, batch, R, n_row_tiles, n_tiles, row_is_state ? 1 : 0, mask, next, list, fuse);
}

template <bool STACK, int MODE>
cudaError_t launch_step_n(const StepView& v, const LaunchEnv& env, const int32_t* states, const uint64_t* stacks,
                          int32_t batch, bool row_is_state, uint32_t* mask, int32_t* next, const RowList& list,
                          const FuseArgs& fuse, cudaStream_t st) {
    if (next)
        return launch_step_t<STACK, MODE, true>(v, env, states, stacks, batch, row_is_state, mask, next, list, fuse,
                                                st);
    return launch_step_t<STACK, MODE, false>(v, env, states, stacks, batch, row_is_state, mask, next, list, fuse, st);
}

template <bool STACK>
cudaError_t launch_step_s(const StepView& v, const LaunchEnv& env, int mode, const int32_t* states,
                          const uint64_t* stacks, int32_t batch, bool row_is_state, uint32_t* mask, int32_t* next,
                          const RowList& list, const FuseArgs& fuse, cudaStream_t st) {
    switch (mode) {
        case kDenseSmem:
            return launch_step_n<STACK, kDenseSmem>(v, env, states, stacks, batch, row_is_state, mask, next, list, fuse, st);
        case kSparse32Smem:
            return launch_step_n<STACK, kSparse32Smem>(v, env, states, stacks, batch, row_is_state, mask, next, list, fuse, st);
        case kSparse64Smem:
            return launch_step_n<STACK, kSparse64Smem>(v, env, states, stacks, batch, row_is_state, mask, next, list, fuse, st);
        default:
            return launch_step_n<STACK, kDenseGlobal>(v, env, states, stacks, batch, row_is_state, mask, next, list, fuse, st);
    }
}

// Resident CTAs per SM of one kernel, cached per (kernel, device).
int occupancy(const void* kern, int threads) {
    struct Entry {
        const void* fn;
        int dev, n;
    };
    static Entry cache[64];
    static int used = 0;
    static std::mutex mu;   // handles on different host threads share the cache
    int dev = 0;
    cudaGetDevice(&dev);
    {
        std::lock_guard<std::mutex> lk(mu);
        for (int i = 0; i < used; i++)
            if (cache[i].fn == kern && cache[i].dev == dev) return cache[i].n;
    }
    int n = 1;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, threads, 0) != cudaSuccess || n < 1) {
        cudaGetLastError();
        n = 1;
    }
    std::lock_guard<std::mutex> lk(mu);
    if (used < 64) cache[used++] = Entry{kern, dev, n};
    return n;
}

// the gather kernels' dynamic shared memory passes the default 48 KB at 16
// warps: the limit is raised once per device and fold
template <int FOLD>
cudaError_t gather_smem_ready() {
    static bool configured[kMaxDevices] = {false};   // one array per fold
    static std::mutex mu;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return cudaGetLastError();
    if (dev >= kMaxDevices) dev = kMaxDevices - 1;
    std::lock_guard<std::mutex> lk(mu);
    if (!configured[dev]) {
        cudaError_t e = cudaFuncSetAttribute(logits_gather_kernel<FOLD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kGatherMaxWarps * kGatherWarpSmem);
        if (e != cudaSuccess) return e;
        configured[dev] = true;
    }
    return cudaSuccess;
}

}  // namespace

cudaError_t prepare_logits_kernels() {
    cudaError_t e = gather_smem_ready<kFoldLse>();
    if (e == cudaSuccess) e = gather_smem_ready<kFoldMax>();
    if (e == cudaSuccess) e = gather_smem_ready<kFoldSample>();
    return e;
}

namespace {

template <bool BF16, bool STAGE>
cudaError_t launch_logits_t(const LaunchEnv& env, const void* logits, int32_t batch, int64_t stride, int32_t V,
                            const MaskRows& mask, int32_t* argmax, float* lse, float* logprobs, float4* partials,
                            uint32_t* counters, float* lse_tmp, bool out_vec, const SampleArgs* sample,
                            const RowList& list, cudaStream_t st) {
    const int W = (V + 31) / 32;
    const size_t esz = BF16 ? 2 : 4;
    const SampleArgs sa = sample ? *sample : SampleArgs{0u, 0u, 0u, 0u, 1.0f};
    auto reduce = sample ? logits_reduce_kernel<BF16, STAGE, kFoldSample>
                         : (lse || logprobs) ? logits_reduce_kernel<BF16, STAGE, kFoldLse>
                                             : logits_reduce_kernel<BF16, STAGE, kFoldMax>;
    for (int32_t r0 = 0; r0 < batch; r0 += kMaxLogitRows) {
        const int rows = min(kMaxLogitRows, batch - r0);
        // a row list addresses batch rows itself: logits and outputs stay unshifted
        const size_t shift = list.ids ? 0 : (size_t)r0;
        const void* lg = reinterpret_cast<const char*>(logits) + shift * stride * esz;
        MaskRows mk = mask;
        if (mk.row_state) mk.row_state += r0;
        else if (mk.base) mk.base += (size_t)r0 * W;
        RowList lst = list;
        lst.base = r0;
        float* lse_rows = lse ? lse + shift : (logprobs ? lse_tmp : nullptr);
        const long long N = (long long)rows * W;
        // at least 4 batches of 32 words per warp; a pass too small to fill the
        // GPU that way gives each warp fewer (down to one batch) instead
        const int slots = env.num_sms * occupancy((const void*)reduce, kReduceThreads);
        int grid = (int)std::min<long long>((long long)slots, (N + 127) / 128);
        if (grid < slots) grid = (int)std::min<long long>((long long)slots, (N + 31) / 32);
        grid = max(grid, 1);
        long long per_cta = (N + grid - 1) / grid;
        per_cta = std::max<long long>(per_cta, ((long long)W + kMaxSegments - 3) / (kMaxSegments - 2));
        grid = (int)((N + per_cta - 1) / per_cta);
        cudaError_t e0;
        // the gather takes one CTA per row: used when the rows alone fill the
        // SMs (with fewer rows the flat split over rows x words keeps more
        // warps busy)
        if (BF16 && STAGE && rows > env.num_sms) {
            auto gather = sample ? logits_gather_kernel<kFoldSample>
                                 : (lse || logprobs) ? logits_gather_kernel<kFoldLse> : logits_gather_kernel<kFoldMax>;
            // a warp per span of the row, at most kGatherMaxWarps (two CTAs per
            // SM); a warp's words rounded up to whole lanes
            const int nwarps =
                std::max(1, std::min(kGatherMaxWarps, (W + 32 * kGatherSpan - 1) / (32 * kGatherSpan)));
            int chunk = (W + nwarps - 1) / nwarps;
            chunk = (chunk + kGatherSpan - 1) / kGatherSpan * kGatherSpan;
            const int smem = nwarps * kGatherWarpSmem;
            if (cudaError_t e = sample ? gather_smem_ready<kFoldSample>()
                                       : (lse || logprobs) ? gather_smem_ready<kFoldLse>() : gather_smem_ready<kFoldMax>();
                e != cudaSuccess)
                return e;
            e0 = launch_pdl(gather, dim3((unsigned)rows), dim3(nwarps * 32), (size_t)smem, st, lg, stride, mk, V, W,
                            rows, chunk, argmax + shift, lse_rows, sa, (int)shift, logprobs ? 1 : 0, lst);
        } else {
            // a sampling pass draws row r of this chunk with counter row r0 + r
            e0 = launch_pdl(reduce, dim3(grid), dim3(kReduceThreads), 0, st, lg, stride, mk, V, W, rows, per_cta,
                            partials, counters, argmax + shift, lse_rows, sa, (int)shift, lst);
        }
        if (e0 != cudaSuccess) return e0;
        if (logprobs) {
            const long long n_items = (out_vec && STAGE) ? (long long)rows * (V % 16 == 0 ? V / 16 : V / 4) : N;
            int g2 = env.num_sms * occupancy((const void*)logprobs_kernel<BF16, true>, kLogitThreads);
            g2 = (int)std::max<long long>(1, std::min<long long>((long long)g2,
                                                                 (n_items + kLogitThreads - 1) / kLogitThreads));
            // 32-byte vector loads and stores where rows start on 32-byte boundaries
            float* lp = logprobs + (size_t)r0 * V;
            const int wide = (reinterpret_cast<uintptr_t>(lg) % 32 == 0) && ((size_t)stride * esz) % 32 == 0 &&
                             (reinterpret_cast<uintptr_t>(lp) % 32 == 0) && V % 16 == 0;
            cudaError_t e1 = (out_vec && STAGE)
                                 ? launch_pdl(logprobs_kernel<BF16, true>, dim3(g2), dim3(kLogitThreads), 0, st, lg,
                                              stride, mk, V, W, rows, (const float*)lse_rows, lp, wide)
                                 : launch_pdl(logprobs_kernel<BF16, false>, dim3(g2), dim3(kLogitThreads), 0, st, lg,
                                              stride, mk, V, W, rows, (const float*)lse_rows, lp, 0);
            if (e1 != cudaSuccess) return e1;
        }
    }
    return cudaSuccess;
}

}  // namespace

int64_t table_smem_bytes(const StepView& v, bool stack, int mode) {
    const int64_t esz = stack ? 4 : 2;
    const int64_t ret = align16(v.n_ret * 8);
    switch (mode) {
        case kDenseSmem: return align16((int)((int64_t)v.Q * v.K * esz)) + ret;
        case kSparse32Smem: return align16(v.Q * 8) + align16((int)(v.sp_nnz * esz)) + ret;
        case kSparse64Smem: return align16(v.Q * 16) + align16((int)(v.sp_nnz * esz)) + ret;
        default: return 0;
    }
}

int step_fixed_smem_bytes(const StepView& v, bool next) {
    return step_layout(v.K, next ? kRowsPerTileNext : kMaxRowsPerTile, next, v.t32 != nullptr, v.Q, 0,
                       v.self_mask != nullptr)
        .total;
}

cudaError_t launch_step_mask(const StepView& v, const LaunchEnv& env, bool stack, int mode, const int32_t* states,
                             const uint64_t* stacks, int32_t batch, bool row_is_state, uint32_t* mask,
                             int32_t* next, cudaStream_t st, const int32_t* row_ids, const int32_t* row_count,
                             const void* fuse_logits, int64_t fuse_stride, float4* fuse_part, bool fuse_prefetch) {
    const RowList list{row_ids, row_count, 0};
    const FuseArgs fuse{fuse_logits, fuse_stride, fuse_part, fuse_logits && fuse_prefetch ? 1 : 0};
    if (stack)
        return launch_step_s<true>(v, env, mode, states, stacks, batch, row_is_state, mask, next, list, fuse, st);
    return launch_step_s<false>(v, env, mode, states, stacks, batch, row_is_state, mask, next, list, fuse, st);
}

// Merges each row's per-window partials of the fused step: one warp per row.
// ADV: lane 0 then advances the row by its argmax (C.update of the same step).
struct AdvanceArgs {
    const int32_t* states;
    const uint64_t* stacks;
    int32_t* states_out;   // nullptr: no update
    uint64_t* stacks_out;
};

template <bool ADV, bool STACK, int MODE>
__global__ void __launch_bounds__(kLogitThreads)
    fused_combine_kernel(const StepView v, const float4* __restrict__ part, int32_t batch, int32_t n_windows,
                         int32_t* __restrict__ argmax, float* __restrict__ lse, const AdvanceArgs adv) {
    pdl_wait();
    pdl_trigger();
    const int r = blockIdx.x * (kLogitThreads / 32) + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (r >= batch) return;
    float m = -INFINITY, s = 0.0f;
    int idx = INT_MAX;
    for (int k = lane; k < n_windows; k += 32) {
        const float4 p = __ldcg(part + (size_t)r * n_windows + k);
        acc_merge(m, idx, s, p.x, __float_as_int(p.y), p.z);
    }
    warp_merge(m, idx, s);
    if (lane == 0) {
        const int32_t t = m == -INFINITY ? -1 : idx;
        argmax[r] = t;
        if (lse) lse[r] = m == -INFINITY ? -INFINITY : m + logf(s);
        if constexpr (ADV) advance_row<STACK, MODE>(v, adv.states, adv.stacks, r, t, adv.states_out, adv.stacks_out);
    }
}

template <bool STACK>
cudaError_t launch_combine_adv(const StepView& v, int mode, const float4* part, int32_t batch, int32_t n_windows,
                               int32_t* argmax, float* lse, const AdvanceArgs& adv, dim3 grid, cudaStream_t st) {
    switch (mode) {
        case kSparse32Smem:
            return launch_pdl(fused_combine_kernel<true, STACK, kSparse32Smem>, grid, dim3(kLogitThreads), 0, st, v,
                              part, batch, n_windows, argmax, lse, adv);
        case kSparse64Smem:
            return launch_pdl(fused_combine_kernel<true, STACK, kSparse64Smem>, grid, dim3(kLogitThreads), 0, st, v,
                              part, batch, n_windows, argmax, lse, adv);
        default:
            return launch_pdl(fused_combine_kernel<true, STACK, kDenseGlobal>, grid, dim3(kLogitThreads), 0, st, v,
                              part, batch, n_windows, argmax, lse, adv);
    }
}

cudaError_t launch_fused_combine(const StepView& v, bool stack, int mode, const float4* part, int32_t batch,
                                 int32_t n_windows, int32_t* argmax, float* lse, const int32_t* states,
                                 const uint64_t* stacks, int32_t* states_out, uint64_t* stacks_out, cudaStream_t st) {
    const dim3 grid((unsigned)((batch + kLogitThreads / 32 - 1) / (kLogitThreads / 32)));
    const AdvanceArgs adv{states, stacks, states_out, stacks_out};
    if (!states_out)
        return launch_pdl(fused_combine_kernel<false, false, kDenseGlobal>, grid, dim3(kLogitThreads), 0, st, v, part,
                          batch, n_windows, argmax, lse, adv);
    if (stack) return launch_combine_adv<true>(v, mode, part, batch, n_windows, argmax, lse, adv, grid, st);
    return launch_combine_adv<false>(v, mode, part, batch, n_windows, argmax, lse, adv, grid, st);
}

cudaError_t launch_logprobs_bf16(const LaunchEnv& env, const void* logits, int32_t batch, int64_t row_stride,
                                 int32_t V, const uint32_t* mask, const float* lse, float* logprobs, cudaStream_t st) {
    const int W = (V + 31) / 32;
    const bool out_vec = (reinterpret_cast<uintptr_t>(logprobs) % 16 == 0) && (V % 4 == 0);
    for (int32_t r0 = 0; r0 < batch; r0 += kMaxLogitRows) {
        const int rows = min(kMaxLogitRows, batch - r0);
        const void* lg = reinterpret_cast<const char*>(logits) + (size_t)r0 * row_stride * 2;
        const MaskRows mk{mask + (size_t)r0 * W, nullptr, 0, nullptr};
        const long long n_items = out_vec ? (long long)rows * (V % 16 == 0 ? V / 16 : V / 4) : (long long)rows * W;
        int g = env.num_sms * occupancy((const void*)logprobs_kernel<true, true>, kLogitThreads);
        g = (int)std::max<long long>(1, std::min<long long>((long long)g, (n_items + kLogitThreads - 1) / kLogitThreads));
        float* lp = logprobs + (size_t)r0 * V;
        const int wide = (reinterpret_cast<uintptr_t>(lg) % 32 == 0) && ((size_t)row_stride * 2) % 32 == 0 &&
                         (reinterpret_cast<uintptr_t>(lp) % 32 == 0) && V % 16 == 0;
        cudaError_t e = out_vec ? launch_pdl(logprobs_kernel<true, true>, dim3(g), dim3(kLogitThreads), 0, st, lg,
                                             row_stride, mk, V, W, rows, lse + r0, lp, wide)
                                : launch_pdl(logprobs_kernel<true, false>, dim3(g), dim3(kLogitThreads), 0, st, lg,
                                             row_stride, mk, V, W, rows, lse + r0, lp, 0);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

cudaError_t launch_mask_logits(const LaunchEnv& env, const void* logits, int dtype, int32_t batch,
                               int64_t row_stride, int32_t V, const uint32_t* mask, int32_t* argmax, float* lse,
                               float* logprobs, float4* partials, uint32_t* counters, float* lse_tmp,
                               cudaStream_t st, const int32_t* row_state, int32_t Q, uint32_t* err,
                               const SampleArgs* sample, const int32_t* row_ids, const int32_t* row_count) {
    const MaskRows mr{mask, row_state, Q, err};
    const RowList list{row_ids, row_count, 0};
    const bool bf16 = dtype == DOMINO_DTYPE_BF16;
    const bool out_vec = logprobs && (reinterpret_cast<uintptr_t>(logprobs) % 16 == 0) && (V % 4 == 0);
    if (bf16) {
        const bool stage = (reinterpret_cast<uintptr_t>(logits) % 16 == 0) && ((size_t)row_stride * 2) % 16 == 0;
        if (stage)
            return launch_logits_t<true, true>(env, logits, batch, row_stride, V, mr, argmax, lse, logprobs,
                                               partials, counters, lse_tmp, out_vec, sample, list, st);
        return launch_logits_t<true, false>(env, logits, batch, row_stride, V, mr, argmax, lse, logprobs, partials,
                                            counters, lse_tmp, out_vec, sample, list, st);
    }
    return launch_logits_t<false, false>(env, logits, batch, row_stride, V, mr, argmax, lse, logprobs, partials,
                                         counters, lse_tmp, out_vec, sample, list, st);
}

cudaError_t launch_mask_sample(const LaunchEnv& env, const void* logits, int dtype, int32_t batch,
                               int64_t row_stride, int32_t V, const uint32_t* mask, float temperature,
                               uint64_t seed, uint64_t offset, int32_t* tokens, float4* partials,
                               uint32_t* counters, cudaStream_t st) {
    const SampleArgs sa{(uint32_t)seed, (uint32_t)(seed >> 32), (uint32_t)offset, (uint32_t)(offset >> 32),
                        1.0f / temperature};   // one correctly rounded fp32 division
    return launch_mask_logits(env, logits, dtype, batch, row_stride, V, mask, tokens, nullptr, nullptr, partials,
                              counters, nullptr, st, nullptr, 0, nullptr, &sa);
}

// The table image of `mode` staged in shared memory (the step kernel's image:
// dense [Q][K] then pop targets, or the sparse rows, entries, pop targets);
// kDenseGlobal reads the dense image from global memory.
template <bool STACK, int MODE>
cudaError_t launch_advance_m(const StepView& v, const int32_t* states, const uint64_t* stacks, const int32_t* tokens,
                             int32_t batch, int32_t* states_out, uint64_t* stacks_out, cudaStream_t st) {
    const unsigned grid = (unsigned)((batch + kAdvanceThreads - 1) / kAdvanceThreads);
    const uint4* img = nullptr;
    int bytes = 0, tgt_off = 0, ret_off = 0;
    if constexpr (MODE != kDenseGlobal) {
        const size_t esz = STACK ? 4 : 2;
        bytes = (int)table_smem_bytes(v, STACK, MODE);
        if (MODE == kDenseSmem) {
            img = reinterpret_cast<const uint4*>(STACK ? (const void*)v.t32 : (const void*)v.t16);
            ret_off = align16((int)((size_t)v.Q * v.K * esz));
        } else {
            img = reinterpret_cast<const uint4*>(v.sp_info);
            tgt_off = align16(v.Q * (MODE == kSparse32Smem ? 8 : 16));
            ret_off = tgt_off + align16((int)((size_t)v.sp_nnz * esz));
        }
        static int configured[kMaxDevices] = {0};
        static std::mutex mu;
        int dev = 0;
        cudaGetDevice(&dev);
        if (bytes > 48 * 1024 && dev < kMaxDevices) {
            std::lock_guard<std::mutex> lk(mu);
            if (configured[dev] < bytes) {
                cudaError_t e =
                    cudaFuncSetAttribute(advance_kernel<STACK, MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
                if (e != cudaSuccess) return e;
                configured[dev] = bytes;
            }
        }
    }
    return launch_pdl(advance_kernel<STACK, MODE>, dim3(grid), dim3(kAdvanceThreads), (size_t)bytes, st, v, img,
                      bytes / 16, tgt_off, ret_off, states, stacks, tokens, batch, states_out, stacks_out);
}

template <bool STACK>
cudaError_t launch_advance_s(const StepView& v, int mode, const int32_t* states, const uint64_t* stacks,
                             const int32_t* tokens, int32_t batch, int32_t* states_out, uint64_t* stacks_out,
                             cudaStream_t st) {
    switch (mode) {
        case kDenseSmem:
            return launch_advance_m<STACK, kDenseSmem>(v, states, stacks, tokens, batch, states_out, stacks_out, st);
        case kSparse32Smem:
            return launch_advance_m<STACK, kSparse32Smem>(v, states, stacks, tokens, batch, states_out, stacks_out, st);
        case kSparse64Smem:
            return launch_advance_m<STACK, kSparse64Smem>(v, states, stacks, tokens, batch, states_out, stacks_out, st);
        default:
            return launch_advance_m<STACK, kDenseGlobal>(v, states, stacks, tokens, batch, states_out, stacks_out, st);
    }
}

cudaError_t launch_advance(const StepView& v, bool stack, int mode, const int32_t* states, const uint64_t* stacks,
                           const int32_t* tokens, int32_t batch, int32_t* states_out, uint64_t* stacks_out,
                           cudaStream_t st) {
    if (stack) return launch_advance_s<true>(v, mode, states, stacks, tokens, batch, states_out, stacks_out, st);
    return launch_advance_s<false>(v, mode, states, stacks, tokens, batch, states_out, stacks_out, st);
}

cudaError_t launch_advance_table(const int32_t* table_next, int32_t Q, int32_t V, int32_t eos_id, int32_t start,
                                 const int32_t* states, const int32_t* tokens, int32_t batch, int32_t* states_out,
                                 uint32_t* err, cudaStream_t st) {
    const unsigned grid = (unsigned)((batch + kAdvanceThreads - 1) / kAdvanceThreads);
    return launch_pdl(advance_table_kernel, dim3(grid), dim3(kAdvanceThreads), 0, st, table_next, Q, V, eos_id, start,
                      states, tokens, batch, states_out, err);
}


cudaError_t launch_propose_check(const StepView& v, bool stack, int mode, const int32_t* states,
                                 const uint64_t* stacks, const int32_t* proposals, int32_t batch, int32_t* tokens_out,
                                 int32_t* row_ids, int32_t* row_count, cudaStream_t st) {
    const unsigned grid = (unsigned)((batch + kAdvanceThreads - 1) / kAdvanceThreads);
    auto pick = [&](auto kern) {
        return launch_pdl(kern, dim3(grid), dim3(kAdvanceThreads), 0, st, v, states, stacks, proposals, batch,
                          tokens_out, row_ids, row_count);
    };
    if (stack) {
        if (mode == kSparse32Smem) return pick(propose_check_kernel<true, kSparse32Smem>);
        if (mode == kSparse64Smem) return pick(propose_check_kernel<true, kSparse64Smem>);
        return pick(propose_check_kernel<true, kDenseGlobal>);
    }
    if (mode == kSparse32Smem) return pick(propose_check_kernel<false, kSparse32Smem>);
    if (mode == kSparse64Smem) return pick(propose_check_kernel<false, kSparse64Smem>);
    return pick(propose_check_kernel<false, kDenseGlobal>);
}

cudaError_t launch_spec_update(const StepView& v, bool stack, const int32_t* states, const uint64_t* stacks,
                               const int32_t* tokens, int32_t batch, uint32_t* counts, unsigned long long* best,
                               uint32_t* reached, cudaStream_t st) {
    const unsigned grid = (unsigned)((batch + kAdvanceThreads - 1) / kAdvanceThreads);
    if (stack)
        return launch_pdl(spec_update_kernel<true>, dim3(grid), dim3(kAdvanceThreads), 0, st, v, states, stacks,
                          tokens, batch, counts, best, reached);
    return launch_pdl(spec_update_kernel<false>, dim3(grid), dim3(kAdvanceThreads), 0, st, v, states, stacks, tokens,
                      batch, counts, best, reached);
}

cudaError_t launch_spec_propose(const StepView& v, bool stack, int mode, const int32_t* states,
                                const uint64_t* stacks, int32_t batch, int32_t s, int32_t min_permille,
                                const unsigned long long* best, const uint32_t* reached, int32_t* proposals,
                                int32_t* n_prop, int32_t* chain_states, uint64_t* chain_stacks, cudaStream_t st) {
    const unsigned grid = (unsigned)((batch + kAdvanceThreads - 1) / kAdvanceThreads);
    auto pick = [&](auto kern) {
        return launch_pdl(kern, dim3(grid), dim3(kAdvanceThreads), 0, st, v, states, stacks, batch, s, min_permille,
                          best, reached, proposals, n_prop, chain_states, chain_stacks);
    };
    if (stack) {
        if (mode == kSparse32Smem) return pick(spec_propose_kernel<true, kSparse32Smem>);
        if (mode == kSparse64Smem) return pick(spec_propose_kernel<true, kSparse64Smem>);
        return pick(spec_propose_kernel<true, kDenseGlobal>);
    }
    if (mode == kSparse32Smem) return pick(spec_propose_kernel<false, kSparse32Smem>);
    if (mode == kSparse64Smem) return pick(spec_propose_kernel<false, kSparse64Smem>);
    return pick(spec_propose_kernel<false, kDenseGlobal>);
}

cudaError_t launch_spec_accept(const int32_t* proposals, const int32_t* n_prop, const int32_t* decoded,
                               const int32_t* chain_states, const uint64_t* chain_stacks, int32_t batch, int32_t s,
                               int32_t* n_accept, int32_t* tokens_out, int32_t* states_out, uint64_t* stacks_out,
                               cudaStream_t st) {
    const unsigned grid = (unsigned)((batch + kAdvanceThreads - 1) / kAdvanceThreads);
    return launch_pdl(spec_accept_kernel, dim3(grid), dim3(kAdvanceThreads), 0, st, proposals, n_prop, decoded,
                      chain_states, chain_stacks, batch, s, n_accept, tokens_out, states_out, stacks_out);
}

}  // namespace domino

// ---------------------------------------------------------------------------
// domino_mask_logits_noalloc: the masked argmax / log-sum-exp for callers that
// cannot allocate device memory.  Its scratch (per-row partials, tickets and a
// temporary lse) is the fixed array below, part of this library's image, so
// every GPU that loads the library holds it until the process exits.
// ---------------------------------------------------------------------------
namespace {

constexpr int kNoAllocMaxRows = 512;
constexpr int kNoAllocMaxDevices = 64;
constexpr size_t kNoAllocPartialsBytes = sizeof(float4) * (size_t)kNoAllocMaxRows * domino::kMaxSegments;
constexpr size_t kNoAllocCountersBytes = sizeof(uint32_t) * (size_t)kNoAllocMaxRows;
constexpr size_t kNoAllocScratchBytes = kNoAllocPartialsBytes + kNoAllocCountersBytes + sizeof(float) * kNoAllocMaxRows;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];   // 516 KiB

struct NoAllocDevice {
    bool ready;
    unsigned char* scratch;   // device address of g_noalloc_scratch on this device
    int num_sms;
};
NoAllocDevice g_noalloc_dev[kNoAllocMaxDevices];
std::mutex g_noalloc_mu;

// Once per device, with that device current: the array's device address.
int noalloc_setup(int dev, NoAllocDevice* out) {
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    NoAllocDevice& d = g_noalloc_dev[dev];
    if (!d.ready) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) {
            cudaGetLastError();
            return DOMINO_E_CUDA;
        }
        int sms = 0;
        if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1) {
            cudaGetLastError();
            return DOMINO_E_CUDA;
        }
        if (domino::prepare_logits_kernels() != cudaSuccess) {
            cudaGetLastError();
            return DOMINO_E_CUDA;
        }
        d.scratch = static_cast<unsigned char*>(p);
        d.num_sms = sms;
        d.ready = true;
    }
    *out = d;
    return DOMINO_OK;
}

}  // namespace

extern "C" int domino_mask_logits_noalloc(const void* logits_dev, int32_t dtype, int32_t batch, int32_t n_tokens,
                                          int64_t row_stride_elems, const uint32_t* mask_dev, int32_t* argmax_dev,
                                          float* lse_dev, float* logprobs_dev, void* stream) {
    if (dtype != DOMINO_DTYPE_F32 && dtype != DOMINO_DTYPE_BF16) return DOMINO_E_INVALID_ARG;
    if (batch < 0 || batch > kNoAllocMaxRows || n_tokens < 1 || n_tokens > (1 << 24) || row_stride_elems < n_tokens)
        return DOMINO_E_INVALID_ARG;
    if (batch == 0) return DOMINO_OK;
    if (!logits_dev || !mask_dev || !argmax_dev) return DOMINO_E_INVALID_ARG;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return DOMINO_E_CUDA;
    }
    if (dev < 0 || dev >= kNoAllocMaxDevices) return DOMINO_E_UNSUPPORTED;
    NoAllocDevice d{};
    int rc = noalloc_setup(dev, &d);
    if (rc != DOMINO_OK) return rc;
    float4* partials = reinterpret_cast<float4*>(d.scratch);
    uint32_t* counters = reinterpret_cast<uint32_t*>(d.scratch + kNoAllocPartialsBytes);
    float* lse_tmp = reinterpret_cast<float*>(d.scratch + kNoAllocPartialsBytes + kNoAllocCountersBytes);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // the tickets must start at zero; the array keeps whatever the last call left
    cudaError_t e = cudaMemsetAsync(counters, 0, sizeof(uint32_t) * (size_t)batch, st);
    if (e == cudaSuccess) {
        domino::LaunchEnv env{d.num_sms, 0};
        e = domino::launch_mask_logits(env, logits_dev, dtype, batch, row_stride_elems, n_tokens, mask_dev,
                                       argmax_dev, lse_dev, logprobs_dev, partials, counters, lse_tmp, st);
    }
    if (e != cudaSuccess) {
        cudaGetLastError();
        return DOMINO_E_CUDA;
    }
    return DOMINO_OK;
}
