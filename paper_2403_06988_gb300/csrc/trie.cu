// trie.cu -- C.mask() over the prefix tree of the vocabulary (sm_103a).
//
// The mask of a row is the set of tokens whose class string can be walked
// from the row's configuration without reaching the dead state (Alg. 1's
// mask at lookahead k = infinity, Sec. 3.5; EOS iff the state accepts with an
// empty stack).  Walking the prefix tree of all class strings (the
// subterminal tree of Sec. 3.3 / Alg. 2, over byte classes) takes each shared
// prefix's transitions once per row and never enters a subtree whose prefix
// died; it reorders and shares the per-token walks of the plain definition
// without changing their result.
//
// Two kernels (see TrieView for the tree's layout and its batches):
//  tree_clear_kernel  one warp per row: clears the row's mask (and next
//                     states) and sets EOS when the state accepts with an
//                     empty stack.
//  tree_tile_kernel   persistent CTAs, one per SM.  For each of its batches a
//                     CTA stages the batch's walk records (chains of nodes
//                     with one child and no token, walked as one record),
//                     their classes and the units' tokens in shared memory
//                     next to the transition table; then, a block of rows at
//                     a time:
//                       1. each row's configuration at every slot (the upper
//                          nodes the units hang off), by walking the slot's
//                          path from the row's configuration;
//                       2. per slot, the list of rows live there;
//                       3. the emitting slots' (row, token) items, spread over
//                          the CTA; then every (unit, row live at the unit's
//                          slot) pair, one thread each: the thread walks the
//                          unit depth first from the row's configuration,
//                          skipping a record's subtree when the record dies,
//                          with the siblings still to visit on its own stack
//                          (one entry per branching record, at most
//                          kTrieBranch).  A record's tokens set their bits with
//                          global reductions (and store their next state);
//                          so do whole subtrees whose classes all loop on the
//                          row's state (the self-loop skip).
//
// With many rows (the precompute: every state a row) a CTA claims its batches'
// row blocks from a global counter per batch, and a CTA done with its own
// batches stages the batch with the most rows left and claims row blocks from
// it too, so that the CTAs end together.
#include <cuda_runtime.h>

#include <climits>
#include <cstdint>
#include <mutex>

#include "domino_internal.h"
#include "walk_common.cuh"

namespace domino {
namespace {

constexpr int kTileThreads = 1024;
constexpr int kClearThreads = 256;          // 8 warps per CTA
constexpr int kClearSplit = 4;              // warps per row
constexpr int kTrieCfg = 4096;              // (slot, row) configurations per row block
constexpr int kTrieRowBlock = 512;          // most rows per block
constexpr int kTrieMaxDevices = 64;

enum TileCtl : int {
    kCtlUnit = 0,     // (unit, row) pairs claimed in this row block
    kCtlBad = 1,      // a staged record failed its check
    kCtlRow = 2,      // the row block claimed (shared row counters)
    kCtlWords = 4,
};

// Shared-memory layout of the tile kernel (byte offsets).
struct TileLayout {
    int accept, self, table, nodes, sub, cls, toks, units, upre, slots, paths, rowcfg, cfg, lrows, lcount, epre, ctl,
        total;
};

__host__ __device__ inline TileLayout tile_layout(int Q, bool self, bool stack, int table_bytes, const TrieView& tv) {
    TileLayout L{};
    int o = 0;
    L.accept = o;  o += align16(((Q + 31) / 32) * 4);
    L.self = o;    o += self ? align16(Q * 8) : 0;
    L.table = o;   o += align16(table_bytes);
    L.nodes = o;   o += align16(tv.max_nodes * 16);
    L.sub = o;     o += self ? align16(tv.max_nodes * 8) : 0;
    L.cls = o;     o += align16(tv.max_cls);
    L.toks = o;    o += align16(tv.max_toks * 4);
    L.units = o;   o += align16(tv.max_units * 4);
    L.upre = o;    o += align16((tv.max_units + 1) * 4);
    L.slots = o;   o += align16(tv.max_slots * 16);
    L.paths = o;   o += align16(tv.max_slots * tv.max_path);
    L.rowcfg = o;  o += kTrieRowBlock * 16;
    L.cfg = o;     o += kTrieCfg * (stack ? 8 : 4);
    L.lrows = o;   o += kTrieCfg * 2;
    L.lcount = o;  o += align16(kTrieMaxSlots * 4);
    L.epre = o;    o += align16((kTrieMaxSlots + 1) * 4);
    L.ctl = o;     o += kCtlWords * 4;
    L.total = align16(o);
    return L;
}

struct TreeArgs {
    const int32_t* states;
    const uint64_t* stacks;
    int32_t batch;          // rows (the cap of a row list)
    int32_t row_is_state;
    uint32_t* mask;
    int32_t* next;
    int32_t img_bytes, img_tgt_off, img_ret_off;
    int32_t* row_next;      // [batches]: rows claimed of each batch (zero at launch), or nullptr
};

// Sets a mask bit without waiting for the result (a reduction, not an atomic
// that returns the old word).
__device__ __forceinline__ void set_bit(uint32_t* word, uint32_t bit) {
    asm volatile("red.global.or.b32 [%0], %1;" ::"l"(word), "r"(bit) : "memory");
}

// ---------------------------------------------------------------------------
// tree_clear_kernel
// ---------------------------------------------------------------------------
// kClearSplit warps per row, each on a slice of its mask (and next states);
// the warp whose slice holds EOS sets it after clearing.
template <bool NEXT>
__global__ void __launch_bounds__(kClearThreads)
    tree_clear_kernel(const __grid_constant__ StepView v, const __grid_constant__ TreeArgs a, const RowList list) {
    pdl_wait();
    pdl_trigger();
    const int lane = threadIdx.x & 31;
    const int gw = blockIdx.x * (kClearThreads / 32) + (threadIdx.x >> 5);
    const int i = gw / kClearSplit, part = gw - i * kClearSplit;
    if (i >= list.rows(a.batch)) return;
    const int W = v.W, V = v.V, eos = v.eos_id;
    uint32_t* mrow = a.mask ? a.mask + (size_t)i * W : nullptr;
    int32_t* nrow = NEXT && a.next ? a.next + (size_t)i * V : nullptr;
    bool eos_m = false, eos_n = false;   // this warp's slices hold EOS
    if (mrow) {
        const bool vec = (W & 3) == 0 && (reinterpret_cast<uintptr_t>(mrow) & 15) == 0;
        const int n = vec ? W / 4 : W, c = (n + kClearSplit - 1) / kClearSplit;
        const int j0 = part * c, j1 = min(n, j0 + c);
        if (vec) {
            for (int j = j0 + lane; j < j1; j += 32) reinterpret_cast<uint4*>(mrow)[j] = make_uint4(0u, 0u, 0u, 0u);
        } else {
            for (int j = j0 + lane; j < j1; j += 32) mrow[j] = 0u;
        }
        const int e = vec ? (eos >> 5) >> 2 : eos >> 5;
        eos_m = eos >= 0 && e >= j0 && e < j1;
    }
    if (nrow) {
        const bool vec = (V & 3) == 0 && (reinterpret_cast<uintptr_t>(nrow) & 15) == 0;
        const int n = vec ? V / 4 : V, c = (n + kClearSplit - 1) / kClearSplit;
        const int j0 = part * c, j1 = min(n, j0 + c);
        if (vec) {
            for (int j = j0 + lane; j < j1; j += 32) __stcs(reinterpret_cast<int4*>(nrow) + j, make_int4(0, 0, 0, 0));
        } else {
            for (int j = j0 + lane; j < j1; j += 32) nrow[j] = 0;
        }
        const int e = vec ? eos >> 2 : eos;
        eos_n = eos >= 0 && e >= j0 && e < j1;
    }
    __syncwarp();   // the slice is clear before its EOS bit is set
    if (lane == 0 && (part == 0 || eos_m || eos_n)) {
        // the row's configuration (invalid ones set the error word, once per row)
        const int b = list.row(i);
        uint4 rc;
        if (a.row_is_state) {
            const uint32_t q = (uint32_t)b;
            rc = make_uint4(q, 0u, 0u, 1u | (((__ldg(v.accept_bits + (q >> 5)) >> (q & 31u)) & 1u) ? 2u : 0u));
        } else {
            const int32_t sv = __ldg(a.states + b);
            const unsigned long long w =
                a.stacks ? __ldg(reinterpret_cast<const unsigned long long*>(a.stacks) + b) : 0ull;
            rc = decode_row(v, sv, w, a.stacks != nullptr, v.accept_bits, part == 0);
        }
        // EOS: allowed iff the state accepts and the stack is empty; the state stays
        if (rc.w & 2u) {
            if (eos_m) set_bit(mrow + (eos >> 5), 1u << (eos & 31));
            if (eos_n) nrow[eos] = (int32_t)rc.x;
        }
    }
}

// ---------------------------------------------------------------------------
// tree_tile_kernel
// ---------------------------------------------------------------------------
// per-lane configuration packed for shared memory: state | depth << 16 (the
// stack bits apart)
__device__ __forceinline__ uint32_t pack_sd(uint32_t s, uint32_t depth) { return s | (depth << 16); }

template <bool STACK, int MODE, bool NEXT>
struct TileCtx {
    using E = typename std::conditional<STACK, uint32_t, uint16_t>::type;
    const StepView& v;
    const TreeArgs& a;
    const Tab<E, MODE>& tab;
    const uint16_t* ret;
    uint32_t maxd;
    const unsigned long long* s_self;   // nullptr: no self-loop skip
    const uint4* snode;                 // {end | nodes << 16, first token | tokens << 16, first class, 0}
    const uint8_t* scls;                // the records' classes
    const unsigned long long* ssub;
    const int32_t* stok;
    int nn, nt;                         // staged nodes and tokens

    __device__ __forceinline__ void fail() const { atomicOr(v.err, DOMINO_DEVERR_INTERNAL); }

    __device__ __forceinline__ void emit_one(int row, int t, uint32_t s) const {
        if ((uint32_t)t >= (uint32_t)v.V) {   // the tree holds token ids only
            fail();
            return;
        }
        if (a.mask) set_bit(a.mask + (size_t)row * v.W + (t >> 5), 1u << (t & 31));
        if constexpr (NEXT) {
            if (a.next) a.next[(size_t)row * v.V + t] = (int32_t)s;
        }
    }
    // One lane walks unit root x0 for its own row from the configuration
    // (s, bits, depth) at the unit's parent: depth first over the records in
    // preorder, the siblings still to visit on the lane's own stack (one entry
    // per branching record, at most kTrieBranch).
    __device__ __forceinline__ void walk_lane(int row, int x0, uint32_t s, uint32_t bits, uint32_t depth) const {
        int x = x0, end = x0 + 1, sp = 0;
        uint32_t kx[kTrieBranch], ks[kTrieBranch], kb[STACK ? kTrieBranch : 1];
        for (;;) {
            while (x < end) {
                const uint4 rec = snode[x];   // checked when staged
                const int xs = (int)(rec.x & 0xFFFFu), nc = (int)(rec.x >> 16);
                uint32_t b2 = bits, d2 = depth, s2 = s;
                for (int k = 0; k < nc && s2 != 0; ++k)
                    s2 = step_once<STACK>(tab, ret, maxd, s2, scls[rec.z + k], b2, d2);
                if (s2 != 0) {
                    const int tl = (int)(rec.y & 0xFFFFu), ne = (int)(rec.y >> 16);
                    for (int j = tl; j < tl + ne; ++j) emit_one(row, stok[j], s2);
                    if (xs > x + 1) {   // x has children
                        bool desc = true;
                        if (s_self && (ssub[x] & ~s_self[s2]) == 0ull) {
                            // every class below keeps the state: the whole
                            // subtree is allowed with it
                            const int th = xs < nn ? (int)(snode[xs].y & 0xFFFFu) : nt;   // the subtree's tokens end
                            for (int j = tl + ne; j < th; ++j) emit_one(row, stok[j], s2);
                            desc = false;
                        }
                        if (desc) {
                            if (xs < end) {
                                if (sp == kTrieBranch) {   // the tree bounds the stack by kTrieBranch
                                    fail();
                                    return;
                                }
                                kx[sp] = (uint32_t)xs | ((uint32_t)end << 16);
                                ks[sp] = pack_sd(s, depth);
                                if constexpr (STACK) kb[sp] = bits;
                                ++sp;
                            }
                            end = xs;
                            s = s2;
                            bits = b2;
                            depth = d2;
                            x = x + 1;
                            continue;
                        }
                    }
                }
                x = xs;
            }
            if (sp == 0) return;
            --sp;
            x = (int)(kx[sp] & 0xFFFFu);
            end = (int)(kx[sp] >> 16);
            s = ks[sp] & 0xFFFFu;
            depth = ks[sp] >> 16;
            if constexpr (STACK) bits = kb[sp];
        }
    }
};

// The rows per block of a batch with `ns` slots.
__device__ __forceinline__ int rows_per_block(int ns) { return max(1, min(kTrieRowBlock, kTrieCfg / max(ns, 1))); }

// The batch with the most rows left (ties: the lowest index), if at least two
// of its row blocks are left; -1 otherwise.  Every thread of the CTA calls it;
// red holds 33 ints of scratch.
__device__ __forceinline__ int pick_batch(const TrieView& tv, const int32_t* row_next, int nrows, int* red, int tid) {
    const int nb = __ldg(tv.cta_batch + tv.grid);
    unsigned best = 0u;   // rows left << 16 | (0xFFFF - batch)
    for (int b = tid; b < nb; b += kTileThreads) {
        const int taken = *reinterpret_cast<const volatile int32_t*>(row_next + b);
        const uint4 bB = __ldg(tv.batch + 2 * b + 1);
        const int rem = nrows - min(nrows, max(taken, 0));
        if (rem >= 2 * rows_per_block((int)(bB.y - bB.x)))
            best = max(best, ((unsigned)rem << 16) | (0xFFFFu - (unsigned)b));
    }
    best = __reduce_max_sync(0xffffffffu, best);
    __syncthreads();   // red is free
    if ((tid & 31) == 0) red[tid >> 5] = (int)best;
    __syncthreads();
    if (tid < 32) {
        const unsigned w = __reduce_max_sync(0xffffffffu, (unsigned)red[tid]);
        if (tid == 0) red[32] = w == 0u ? -1 : (int)(0xFFFFu - (w & 0xFFFFu));
    }
    __syncthreads();
    return red[32];
}

// 1024 threads a CTA: at most 64 registers a thread.  STEAL: row blocks
// claimed from a.row_next, other CTAs' batches taken once a CTA's own are done.
template <bool STACK, int MODE, bool NEXT, bool STEAL>
__global__ void __maxnreg__(64)
    tree_tile_kernel(const __grid_constant__ StepView v, const __grid_constant__ TrieView tv,
                     const uint4* __restrict__ img, const __grid_constant__ TreeArgs a, const RowList list) {
    using E = typename std::conditional<STACK, uint32_t, uint16_t>::type;
    extern __shared__ __align__(16) unsigned char smem[];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const bool use_self = v.self_mask != nullptr;
    const TileLayout L = tile_layout(v.Q, use_self, STACK, MODE == kDenseGlobal ? 0 : a.img_bytes, tv);
    uint32_t* s_accept = reinterpret_cast<uint32_t*>(smem + L.accept);
    unsigned long long* s_self = reinterpret_cast<unsigned long long*>(smem + L.self);
    // a staged walk record: {end record | nodes << 16, first token | tokens << 16, first class, 0}
    uint4* snode = reinterpret_cast<uint4*>(smem + L.nodes);
    uint8_t* scls = reinterpret_cast<uint8_t*>(smem + L.cls);
    unsigned long long* ssub = reinterpret_cast<unsigned long long*>(smem + L.sub);
    int32_t* stok = reinterpret_cast<int32_t*>(smem + L.toks);
    uint32_t* sunit = reinterpret_cast<uint32_t*>(smem + L.units);   // root - nb | slot << 16
    int* upre = reinterpret_cast<int*>(smem + L.upre);               // the units' first (row, unit) pairs
    uint4* sslot = reinterpret_cast<uint4*>(smem + L.slots);         // {path length, 0, first token, tokens set}
    uint8_t* spath = reinterpret_cast<uint8_t*>(smem + L.paths);
    uint4* rowcfg = reinterpret_cast<uint4*>(smem + L.rowcfg);
    uint32_t* cfg = reinterpret_cast<uint32_t*>(smem + L.cfg);       // [slot][row] state | depth << 16 (+ bits)
    uint16_t* lrows = reinterpret_cast<uint16_t*>(smem + L.lrows);   // [slot][k] live rows of the block
    int* lcount = reinterpret_cast<int*>(smem + L.lcount);
    int* epre = reinterpret_cast<int*>(smem + L.epre);   // the emitting slots' first (row, token) items
    int* ctl = reinterpret_cast<int*>(smem + L.ctl);
    const int b0 = __ldg(tv.cta_batch + blockIdx.x), b1 = __ldg(tv.cta_batch + blockIdx.x + 1);
    if (b0 >= b1 && !STEAL) {   // no units for this CTA
        pdl_wait();
        return;
    }
    for (int i = tid; i < (v.Q + 31) / 32; i += kTileThreads) s_accept[i] = __ldg(v.accept_bits + i);
    if (use_self)
        for (int i = tid; i < v.Q; i += kTileThreads) s_self[i] = __ldg(v.self_mask + i);
    Tab<E, MODE> tab;
    tab.K = (uint32_t)v.K;
    debug_bounds(tab, v);
    const uint16_t* ret;
    if constexpr (MODE == kDenseGlobal) {
        tab.dense = reinterpret_cast<const E*>(STACK ? (const void*)v.t32 : (const void*)v.t16);
        ret = v.ret;
    } else {
        uint4* dst = reinterpret_cast<uint4*>(smem + L.table);
        for (int i = tid; i < a.img_bytes / 16; i += kTileThreads) dst[i] = __ldg(img + i);
        const unsigned char* t = smem + L.table;
        tab.dense = reinterpret_cast<const E*>(t);
        tab.sp = reinterpret_cast<const uint32_t*>(t);
        tab.tgt = reinterpret_cast<const E*>(t + a.img_tgt_off);
        ret = reinterpret_cast<const uint16_t*>(t + a.img_ret_off);
    }
    const uint32_t maxd = (uint32_t)v.max_depth;
    bool waited = false;
    for (int own = b0;;) {
        int bj = own;
        if (own < b1) {
            ++own;
        } else {
            if constexpr (!STEAL) break;
            if (!waited) {   // the row counters are zeroed before the clear kernel
                pdl_wait();
                waited = true;
            }
            bj = pick_batch(tv, a.row_next, list.rows(a.batch), lcount, tid);
            if (bj < 0) break;
        }
        const uint4 bA = __ldg(tv.batch + 2 * bj);       // units [x, y), ranges [z, w)
        const uint4 bB = __ldg(tv.batch + 2 * bj + 1);   // slots [x, y), staged nodes z, tokens w
        const int nk = (int)(bA.y - bA.x), nn = (int)bB.z, nt = (int)bB.w;
        const int ns = (int)(bB.y - bB.x);
        __syncthreads();   // the previous batch is done with shared memory
        if (tid == 0) ctl[kCtlBad] = 0;
        __syncthreads();
        // the batch's record, class and token ranges, staged one after the
        // other; a record's subtree end, first class and first token become
        // staged indices
        int sb = 0, tb = 0, cb = 0;
        for (uint32_t ri = bA.z; ri < bA.w; ++ri) {
            const uint4 R = __ldg(tv.range + 2 * ri);       // {first record, end record, first token, end token}
            const uint4 Rn = __ldg(tv.range + 2 * ri + 1);  // {first node, end node, 0, 0}
            const int rn = (int)(R.y - R.x), rt = (int)(R.w - R.z), rc = (int)(Rn.y - Rn.x);
            if (rn < 0 || rt < 0 || rc < 0 || sb + rn > nn || tb + rt > nt || cb + rc > tv.max_cls) {
                if (tid == 0) ctl[kCtlBad] = 1;
                break;
            }
            for (int n = tid; n < rn; n += kTileThreads) {
                const uint4 r0 = __ldg(tv.node + 2 * ((size_t)R.x + n));
                const uint4 r1 = __ldg(tv.node + 2 * ((size_t)R.x + n) + 1);
                // preorder (a subtree ends after its record), the record's nodes
                // and tokens inside the range's: the walk relies on all three.
                // The upper nodes between a range's units are staged too (never
                // walked); their subtrees end past the range, so skips are
                // clamped to its end.
                const uint32_t xs = min(r0.x - R.x, (uint32_t)rn), tl = r0.w - R.z, fc = r0.y - Rn.x;
                if (xs <= (uint32_t)n || tl > (uint32_t)rt || r1.x > (uint32_t)rt - tl || r0.z == 0u ||
                    r0.z > 255u || fc >= (uint32_t)rc || r0.z > (uint32_t)rc - fc)
                    ctl[kCtlBad] = 1;
                snode[sb + n] = make_uint4((xs + sb) | (min(r0.z, 255u) << 16), (tl + tb) | (r1.x << 16), fc + cb, 0u);
                if (use_self) ssub[sb + n] = ((unsigned long long)r1.z << 32) | r1.y;
            }
            for (int j = tid; j < rc; j += kTileThreads) scls[cb + j] = __ldg(tv.ncls + Rn.x + j);
            for (int j = tid; j < rt; j += kTileThreads) stok[tb + j] = __ldg(tv.dtok + R.z + j);
            sb += rn;
            tb += rt;
            cb += rc;
        }
        if ((sb != nn || tb != nt) && tid == 0) ctl[kCtlBad] = 1;
        for (int k = tid; k < nk; k += kTileThreads) {
            const uint2 un = __ldg(tv.unit + bA.x + k);
            if (un.x >= (uint32_t)nn || un.y >= (uint32_t)ns) ctl[kCtlBad] = 1;
            sunit[k] = un.x | (un.y << 16);
        }
        for (int k = tid; k < ns; k += kTileThreads) {
            const uint4 sl = __ldg(tv.slot + bB.x + k);   // {upper index, first token, tokens set, 0}
            const uint4 up = __ldg(tv.upper + sl.x);      // {node, path offset, path length, 0}
            if (up.z > (uint32_t)tv.max_path) ctl[kCtlBad] = 1;
            sslot[k] = make_uint4(min(up.z, (uint32_t)tv.max_path), 0u, sl.y, sl.z);
            for (uint32_t d = 0; d < up.z && d < (uint32_t)tv.max_path; ++d)
                spath[k * tv.max_path + d] = __ldg(tv.upath + up.y + d);
        }
        if (!waited) {   // everything above is the static tree; the masks come from tree_clear_kernel
            // no early launch of the next kernel: one launched early parks its
            // CTAs beside these, and a logits pass queued that way took about
            // 10 us longer than one launched when this grid ends (GB300, batch
            // 256, V = 128256)
            pdl_wait();
            waited = true;
        }
        __syncthreads();
        if (ctl[kCtlBad]) {   // a record the walk cannot trust: report and skip the batch
            if (tid == 0) atomicOr(v.err, DOMINO_DEVERR_INTERNAL);
            continue;
        }
        const TileCtx<STACK, MODE, NEXT> cx{v, a, tab, ret, maxd, use_self ? s_self : nullptr, snode, scls, ssub, stok,
                                            nn, nt};
        const int nrows = list.rows(a.batch);
        const int rb = rows_per_block(ns);
        for (int r0 = 0;; r0 += rb) {
            if constexpr (STEAL) {   // the previous block ended with a barrier
                if (tid == 0) ctl[kCtlRow] = atomicAdd(a.row_next + bj, rb);
                __syncthreads();
                r0 = ctl[kCtlRow];
            }
            if (r0 >= nrows) break;
            const int nr = min(rb, nrows - r0);
            if (tid < ns) lcount[tid] = 0;
            if (tid == 0) ctl[kCtlUnit] = 0;
            // 1. the rows' configurations
            for (int r = tid; r < nr; r += kTileThreads) {
                const int b = list.row(r0 + r);
                if (a.row_is_state) {
                    rowcfg[r] = make_uint4((uint32_t)b, 0u, 0u, 1u);
                } else {
                    const int32_t sv = __ldg(a.states + b);
                    const unsigned long long w =
                        a.stacks ? __ldg(reinterpret_cast<const unsigned long long*>(a.stacks) + b) : 0ull;
                    rowcfg[r] = decode_row(v, sv, w, a.stacks != nullptr, s_accept, false);
                }
            }
            __syncthreads();
            // ... at every slot: the slot's path from the row's configuration
            for (int f = tid; f < ns * nr; f += kTileThreads) {
                const int k = f / nr, r = f - k * nr;
                const uint4 rc = rowcfg[r];
                uint32_t s = (rc.w & 1u) ? rc.x : 0u, bits = rc.y, depth = rc.z;
                const int plen = (int)sslot[k].x;
                for (int d = 0; d < plen && s != 0; ++d)
                    s = step_once<STACK>(tab, ret, maxd, s, spath[k * tv.max_path + d], bits, depth);
                cfg[f] = pack_sd(s, depth);
                if constexpr (STACK) cfg[kTrieCfg + f] = bits;
            }
            __syncthreads();
            // 2. per slot, the rows live there (a warp's lanes take consecutive
            // rows of one slot: one counter update per warp and slot)
            for (int f0 = warp * 32; f0 < ns * nr; f0 += kTileThreads) {
                const int f = f0 + lane;
                const bool in = f < ns * nr;
                const int k = in ? f / nr : 0, r = in ? f - k * nr : 0;
                const uint32_t sd = in ? cfg[f] : 0u;
                const bool live = in && (sd & 0xFFFFu) != 0u;
                // lanes of the same slot form runs: one atomic per run
                const int k0 = __shfl_sync(0xffffffffu, k, 0);
                const unsigned same = __ballot_sync(0xffffffffu, in && k == k0);
                const unsigned lv = __ballot_sync(0xffffffffu, live);
                int base = 0;
                if (lane == 0 && (lv & same)) base = atomicAdd(&lcount[k0], __popc(lv & same));
                base = __shfl_sync(0xffffffffu, base, 0);
                if (live) {
                    if ((same >> lane) & 1u) {
                        lrows[k0 * rb + base + __popc(lv & same & ((1u << lane) - 1u))] = (uint16_t)r;
                    } else {
                        lrows[k * rb + atomicAdd(&lcount[k], 1)] = (uint16_t)r;
                    }
                }
            }
            __syncthreads();
            // 3. the (unit, live row at the unit's slot) pairs, one lane each:
            // most rows die at the unit's first record, so lanes that walk
            // their own pairs waste far fewer lookups than a warp walking a
            // unit for all its rows in lockstep.  Warp 0 forms the pairs'
            // prefix over the units (a unit's pairs are consecutive).
            if (warp == 1) {
                // emitting slots: (live row, token ending at the slot's node)
                // items, prefix over the slots
                int e0 = 0, e1 = 0;
                if (lane < ns) e0 = lcount[lane] * (int)sslot[lane].w;
                if (lane + 32 < ns) e1 = lcount[lane + 32] * (int)sslot[lane + 32].w;
                int i0 = e0, i1 = e1;
#pragma unroll
                for (int off = 1; off < 32; off <<= 1) {
                    const int y0 = __shfl_up_sync(0xffffffffu, i0, off), y1 = __shfl_up_sync(0xffffffffu, i1, off);
                    if (lane >= off) i0 += y0, i1 += y1;
                }
                const int tot0 = __shfl_sync(0xffffffffu, i0, 31);
                if (lane < ns) epre[lane] = i0 - e0;
                if (lane + 32 < ns) epre[lane + 32] = tot0 + i1 - e1;
                if (lane == 31) epre[ns] = tot0 + (ns > 32 ? i1 : 0);
            }
            if (warp == 0) {
                const int per = (nk + 31) / 32, k0 = lane * per, k1 = min(nk, k0 + per);
                int sum = 0;
                for (int k = k0; k < k1; ++k) sum += lcount[sunit[k] >> 16];
                int incl = sum;
#pragma unroll
                for (int off = 1; off < 32; off <<= 1) {
                    const int y = __shfl_up_sync(0xffffffffu, incl, off);
                    if (lane >= off) incl += y;
                }
                int run = incl - sum;
                for (int k = k0; k < k1; ++k) {
                    upre[k] = run;
                    run += lcount[sunit[k] >> 16];
                }
                if (lane == 31) upre[nk] = incl;
            }
            __syncthreads();
            // the emitting slots' items, spread over the CTA (tokens read from
            // the preorder list in global memory: all loads independent)
            for (int f = tid; f < epre[ns]; f += kTileThreads) {
                int k = 0, hi = ns;   // the slot: epre[k] <= f < epre[k + 1]
                while (hi - k > 1) {
                    const int mid = (k + hi) >> 1;
                    if (epre[mid] <= f) k = mid;
                    else hi = mid;
                }
                const uint4 sl = sslot[k];
                const int g = f - epre[k], nt_k = (int)sl.w;
                const int li = g / nt_k, j = g - li * nt_k;
                const int r = lrows[k * rb + li];
                cx.emit_one(r0 + r, __ldg(tv.dtok + sl.z + j), cfg[k * nr + r] & 0xFFFFu);
            }
            // warps take 32 consecutive pairs at a time (the costliest units'
            // first), so that no warp is left with the last long walks
            const int npairs = upre[nk];
            for (;;) {
                int i = 0;
                if (lane == 0) i = atomicAdd(&ctl[kCtlUnit], 32);
                i = __shfl_sync(0xffffffffu, i, 0) + lane;
                if (i - lane >= npairs) break;
                if (i >= npairs) continue;
                int lo = 0, hi = nk;   // the unit: upre[lo] <= i < upre[lo + 1]
                while (hi - lo > 1) {
                    const int mid = (lo + hi) >> 1;
                    if (upre[mid] <= i) lo = mid;
                    else hi = mid;
                }
                const uint32_t un = sunit[lo];
                const int x0 = (int)(un & 0xFFFFu), sl = (int)(un >> 16);
                const int r = lrows[sl * rb + (i - upre[lo])];
                const uint32_t sd = cfg[sl * nr + r];
                const uint32_t bits = STACK ? cfg[kTrieCfg + sl * nr + r] : 0u;
                cx.walk_lane(r0 + r, x0, sd & 0xFFFFu, bits, sd >> 16);
            }
            __syncthreads();
        }
    }
}

template <typename K>
cudaError_t allow_smem(K kern, int bytes, int* configured, std::mutex& mu) {
    int dev = 0;
    cudaGetDevice(&dev);
    if (bytes <= 48 * 1024 || dev >= kTrieMaxDevices) return cudaSuccess;
    std::lock_guard<std::mutex> lk(mu);
    if (configured[dev] >= bytes) return cudaSuccess;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess) configured[dev] = bytes;
    return e;
}

template <bool STACK, int MODE, bool NEXT>
cudaError_t launch_tree_t(const StepView& v, const TrieView& tv, const LaunchEnv& env, TreeArgs a,
                          const RowList& list, cudaStream_t st) {
    const int img_bytes = MODE == kDenseGlobal ? 0 : (int)table_smem_bytes(v, STACK, MODE);
    a.img_bytes = img_bytes;
    const uint4* img = nullptr;
    a.img_tgt_off = a.img_ret_off = 0;
    if constexpr (MODE != kDenseGlobal) {
        const size_t esz = STACK ? 4 : 2;
        if (MODE == kDenseSmem) {
            img = reinterpret_cast<const uint4*>(STACK ? (const void*)v.t32 : (const void*)v.t16);
            a.img_ret_off = align16((int)((size_t)v.Q * v.K * esz));
        } else {
            img = reinterpret_cast<const uint4*>(v.sp_info);
            a.img_tgt_off = align16(v.Q * (MODE == kSparse32Smem ? 8 : 16));
            a.img_ret_off = a.img_tgt_off + align16((int)((size_t)v.sp_nnz * esz));
        }
    }
    const TileLayout L = tile_layout(v.Q, v.self_mask != nullptr, STACK, img_bytes, tv);
    if (L.total > env.max_smem_optin || tv.max_slots > kTrieMaxSlots || tv.grid > env.num_sms)
        return cudaErrorInvalidConfiguration;
    static std::mutex mu;
    // the precompute (every state a row): shared row counters and stealing
    const bool steal = !STACK && NEXT && a.row_next && a.row_is_state && !list.ids && tv.n_batches > 0 &&
                       tv.n_batches <= 0xFFFF && a.batch <= 0xFFFF;
    if (!steal) a.row_next = nullptr;
    const int clear_grid = (int)(((int64_t)a.batch * kClearSplit + kClearThreads / 32 - 1) / (kClearThreads / 32));
    cudaError_t e = cudaSuccess;
    if constexpr (!STACK && NEXT) {
        if (steal) {
            auto tile = tree_tile_kernel<false, MODE, true, true>;
            static int configured[kTrieMaxDevices] = {0};
            if ((e = allow_smem(tile, L.total, configured, mu)) != cudaSuccess) return e;
            if ((e = cudaMemsetAsync(a.row_next, 0, (size_t)tv.n_batches * 4, st)) != cudaSuccess) return e;
            e = launch_pdl(tree_clear_kernel<NEXT>, dim3(clear_grid), dim3(kClearThreads), 0, st, v, a, list);
            if (e != cudaSuccess) return e;
            return launch_pdl(tile, dim3(tv.grid), dim3(kTileThreads), (size_t)L.total, st, v, tv, img, a, list);
        }
    }
    auto tile = tree_tile_kernel<STACK, MODE, NEXT, false>;
    static int configured[kTrieMaxDevices] = {0};
    if ((e = allow_smem(tile, L.total, configured, mu)) != cudaSuccess) return e;
    e = launch_pdl(tree_clear_kernel<NEXT>, dim3(clear_grid), dim3(kClearThreads), 0, st, v, a, list);
    if (e != cudaSuccess) return e;
    return launch_pdl(tile, dim3(tv.grid), dim3(kTileThreads), (size_t)L.total, st, v, tv, img, a, list);
}

template <bool STACK, bool NEXT>
cudaError_t launch_tree_m(const StepView& v, const TrieView& tv, const LaunchEnv& env, int mode, const TreeArgs& a,
                          const RowList& list, cudaStream_t st) {
    switch (mode) {
        case kDenseSmem: return launch_tree_t<STACK, kDenseSmem, NEXT>(v, tv, env, a, list, st);
        case kSparse32Smem: return launch_tree_t<STACK, kSparse32Smem, NEXT>(v, tv, env, a, list, st);
        case kSparse64Smem: return launch_tree_t<STACK, kSparse64Smem, NEXT>(v, tv, env, a, list, st);
        default: return launch_tree_t<STACK, kDenseGlobal, NEXT>(v, tv, env, a, list, st);
    }
}

}  // namespace

int trie_tile_smem_bytes(const StepView& v, const TrieView& tv, bool stack, int table_bytes) {
    return tile_layout(v.Q, v.self_mask != nullptr, stack, table_bytes, tv).total;
}

cudaError_t launch_trie_step(const StepView& v, const TrieView& tv, const LaunchEnv& env, bool stack, int mode,
                             const int32_t* states, const uint64_t* stacks, int32_t batch, bool row_is_state,
                             uint32_t* mask, int32_t* next, cudaStream_t st, const int32_t* row_ids,
                             const int32_t* row_count, int32_t* row_next) {
    if (batch <= 0) return cudaSuccess;
    TreeArgs a{};
    a.row_next = row_next;
    a.states = states;
    a.stacks = stacks;
    a.batch = batch;
    a.row_is_state = row_is_state ? 1 : 0;
    a.mask = mask;
    a.next = next;
    const RowList list{row_ids, row_count, 0};
    if (stack) {
        return next ? launch_tree_m<true, true>(v, tv, env, mode, a, list, st)
                    : launch_tree_m<true, false>(v, tv, env, mode, a, list, st);
    }
    return next ? launch_tree_m<false, true>(v, tv, env, mode, a, list, st)
                : launch_tree_m<false, false>(v, tv, env, mode, a, list, st);
}

}  // namespace domino
