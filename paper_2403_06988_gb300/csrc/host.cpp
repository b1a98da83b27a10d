// host.cpp -- the C ABI of libdomino.so: handle lifetime, loaders (validation,
// dead-state canonicalisation, byte-class compression, vocabulary arena) and
// argument checks in front of the kernels in kernels.cu.
#include <cuda_runtime.h>

#include <algorithm>
#include <chrono>
#include <cmath>
#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <new>
#include <numeric>
#include <unordered_map>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "domino.h"
#include "domino_internal.h"

using namespace domino;

namespace {

struct DevBuf {
    void* p = nullptr;
    size_t n = 0;
};

}  // namespace

struct domino_ctx {
    int device = -1;
    LaunchEnv env{0, 0};

    // ---- vocabulary (host copy, kept so the arena can be rebuilt per automaton)
    bool vocab_loaded = false;
    int32_t V = 0, W = 0, eos_id = -1, max_len = 0;
    std::vector<uint8_t> tok_bytes;
    std::vector<int64_t> tok_off;

    // ---- automaton (preprocessed)
    bool auto_loaded = false;
    int32_t Q = 0, K = 0, start = 0, max_depth = 0, n_rules = 0;
    bool stack = false;
    uint8_t byte_class[256] = {0};
    std::vector<uint16_t> t16;
    std::vector<uint32_t> t32;
    std::vector<uint16_t> ret;
    std::vector<uint32_t> accept_bits;
    std::vector<uint64_t> self_mask;   // [Q]: classes that keep the state (no stack action); empty if unused
    int32_t sp_nnz = 0;       // live entries of the sparse table (0: no sparse image)
    int32_t sp_words = 0;     // uint32 words per state in the sparse row info (2 or 4)
    int64_t dense_ret_off = 0, sp_tgt_off = 0, sp_ret_off = 0;

    // ---- device copies
    DevBuf d_head, d_info, d_tail_off, d_tail, d_pos_of, d_cls_start, d_eos_slot;
    DevBuf d_dense, d_sparse, d_accept, d_self, d_tok_cls;
    DevBuf d_err, d_partials, d_counters, d_lse_tmp, d_fpart;
    bool arena_ready = false;
    // prefix tree of the class strings and its per-CTA batches (see TrieView)
    DevBuf d_tnode, d_tncls, d_tdtok, d_tupper, d_tupath, d_tbatch, d_trange, d_tslot, d_tunit, d_tcta;
    DevBuf d_trow;                   // the precompute's row counter per batch
    std::vector<uint4> t_node;       // host copies (domino_get_prefix_tree)
    std::vector<uint4> t_cnode;      // the walk's records (chains of nodes), two per record
    std::vector<uint32_t> t_hc;      // [n_nodes + 1]: records before each node
    std::vector<uint8_t> t_ncls;     // each node's class
    std::vector<int32_t> t_dtok;
    std::vector<uint4> t_upper;      // {node, path offset, path length, 0}
    std::vector<uint8_t> t_upath;
    std::vector<uint2> t_unit;       // {root node, parent upper index}
    // per-CTA batches (see TrieView)
    std::vector<uint4> t_batch;      // two per batch
    std::vector<uint4> t_range;      // {first node, end node, first token, end token}
    std::vector<uint4> t_slot;
    std::vector<uint2> t_bunit;      // {root node, slot within the batch}
    std::vector<int32_t> t_cta;      // [grid + 1] first batch of each CTA
    int32_t t_nodes = 0, t_grid = 0;
    int32_t t_max_nodes = 0, t_max_cls = 0, t_max_toks = 0, t_max_units = 0, t_max_slots = 0, t_max_path = 0;
    int t_mode = kDenseGlobal;       // where the tile kernel reads transitions
    bool trie_built = false;         // host arrays valid
    bool trie_ready = false;         // device copies valid
    // which walk the mask step takes: -1 chosen from the automaton (see
    // use_tree), 1 the prefix tree, 0 every token on its own (DOMINO_WALK=tree
    // or =token in the environment when the handle is created)
    int walk_pref = -1;
    int32_t n_windows = 0;
    // staging for domino_decode_step_host
    // s_io packs the step's small inputs and outputs (see io_layout) so that
    // each direction takes one copy through the pinned staging buffer h_io
    DevBuf s_logits, s_mask, s_io;
    void* h_io = nullptr;
    void* h_io_dev = nullptr;   // h_io as the device addresses it
    size_t h_io_n = 0;
    // opportunistic masking: proposals, the fallback row list and its length
    DevBuf o_prop, o_rows, o_count;
    // domino_decode_step_host: a copy stream and the events that hand each
    // chunk of rows from the copies to the kernels
    cudaStream_t cp_stream = nullptr;
    cudaEvent_t ev_cfg = nullptr;
    cudaEvent_t ev_chunk[8] = {};
    cudaEvent_t ev_t[4] = {};       // the chunked copy's start and end (2, 3)
    // host wall time of each path for pinned bf16 logits, a moving average
    // over settled calls: [0] the chunked copy, [1] the in-place read (0: not
    // yet seen)
    double t_wall_ms[2] = {0.0, 0.0};
    // Recorded host-buffer steps: a call whose buffers, sizes and path match an
    // earlier one replays that call's CUDA graph instead of issuing each copy
    // and launch again.  Cleared when an automaton or vocabulary is loaded.
    struct HostGraph {
        const void* key[16];
        cudaGraphExec_t exec;
        uint64_t used;
    };
    std::vector<HostGraph> host_graphs;
    uint64_t host_calls = 0;
};

namespace {

StepView make_view(domino_ctx* h);
int cuda_status(cudaError_t e);

struct DeviceGuard {
    int prev = -1;
    bool changed = false;
    explicit DeviceGuard(int dev) {
        if (dev < 0) return;
        if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) {
            changed = cudaSetDevice(dev) == cudaSuccess;
        }
    }
    ~DeviceGuard() {
        if (changed) cudaSetDevice(prev);
    }
};

void dev_free(DevBuf& b) {
    if (b.p) cudaFree(b.p);
    b.p = nullptr;
    b.n = 0;
}

int64_t dev_bytes(const domino_ctx* h) {
    const DevBuf* all[] = {&h->d_head, &h->d_info, &h->d_tail_off, &h->d_tail, &h->d_pos_of, &h->d_cls_start,
                           &h->d_eos_slot, &h->d_dense, &h->d_sparse, &h->d_accept, &h->d_self, &h->d_tok_cls, &h->d_err, &h->d_fpart, &h->d_partials,
                           &h->d_counters, &h->d_lse_tmp, &h->s_logits, &h->s_mask, &h->s_io,
                           &h->o_prop, &h->o_rows, &h->o_count};
    int64_t n = 0;
    for (auto* b : all) n += (int64_t)b->n;
    return n;
}

// (Re)allocates b to hold n bytes and uploads src (when non-null).
int dev_upload(DevBuf& b, const void* src, size_t n) {
    size_t want = ((n ? n : 16) + 15) / 16 * 16;   // vector staging reads whole 16-byte words
    if (b.n < want) {
        dev_free(b);
        if (cudaMalloc(&b.p, want) != cudaSuccess) {
            cudaGetLastError();
            b.p = nullptr;
            return DOMINO_E_OOM;
        }
        b.n = want;
    }
    if (src && n && cudaMemcpy(b.p, src, n, cudaMemcpyHostToDevice) != cudaSuccess) {
        cudaGetLastError();
        return DOMINO_E_CUDA;
    }
    return DOMINO_OK;
}

int dev_reserve(DevBuf& b, size_t n) { return dev_upload(b, nullptr, n); }

bool is_host_only(const domino_ctx* h) { return h->device < 0; }

void clear_host_graphs(domino_ctx* h) {
    for (auto& g : h->host_graphs) cudaGraphExecDestroy(g.exec);
    h->host_graphs.clear();
    h->t_wall_ms[0] = h->t_wall_ms[1] = 0.0;   // the paths are timed afresh
}

// The prefix tree of the tokens' class strings (TrieView), built from the
// tokens sorted by class string: a token shares with its predecessor the
// nodes of their longest common prefix and opens new nodes for the rest, so
// nodes come out in preorder.  EOS and empty tokens are not in the tree (the
// kernel sets EOS from the row's acceptance; other empty tokens are never
// allowed).  Host arrays only; build_trie uploads them.
void build_trie_host(domino_ctx* h) {
    h->trie_built = h->trie_ready = false;
    h->t_node.clear();
    h->t_cnode.clear();
    h->t_hc.clear();
    h->t_ncls.clear();
    h->t_dtok.clear();
    h->t_upper.clear();
    h->t_upath.clear();
    h->t_unit.clear();
    if (!h->vocab_loaded || !h->auto_loaded) return;
    std::vector<uint8_t> cls(h->tok_bytes.size());
    for (size_t i = 0; i < cls.size(); i++) cls[i] = h->byte_class[h->tok_bytes[i]];
    std::vector<int32_t> order;
    order.reserve((size_t)h->V);
    for (int32_t t = 0; t < h->V; t++)
        if (t != h->eos_id && h->tok_off[t + 1] > h->tok_off[t]) order.push_back(t);
    auto str = [&](int32_t t) { return cls.data() + h->tok_off[t]; };
    auto len = [&](int32_t t) { return (size_t)(h->tok_off[t + 1] - h->tok_off[t]); };
    std::sort(order.begin(), order.end(), [&](int32_t a, int32_t b) {
        const size_t la = len(a), lb = len(b);
        const int c = std::memcmp(str(a), str(b), std::min(la, lb));
        if (c != 0) return c < 0;
        if (la != lb) return la < lb;
        return a < b;
    });
    std::vector<uint32_t> skip, tok_lo, n_end, tok_hi;
    std::vector<uint8_t> ncls;
    std::vector<int32_t> dtok;
    dtok.reserve(order.size());
    std::vector<uint32_t> path;   // open nodes, root first
    auto open_node = [&](uint8_t c) {
        path.push_back((uint32_t)skip.size());
        skip.push_back(0);
        tok_lo.push_back((uint32_t)dtok.size());
        n_end.push_back(0);
        tok_hi.push_back(0);
        ncls.push_back(c);
    };
    auto close_node = [&]() {
        const uint32_t n = path.back();
        path.pop_back();
        skip[n] = (uint32_t)skip.size();
        tok_hi[n] = (uint32_t)dtok.size();
    };
    open_node(0);   // root
    const uint8_t* prev = nullptr;
    size_t prev_len = 0;
    for (int32_t t : order) {
        const uint8_t* s = str(t);
        const size_t L = len(t);
        size_t l = 0;
        while (prev && l < std::min(L, prev_len) && prev[l] == s[l]) l++;
        while (path.size() > l + 1) close_node();
        for (size_t d = l; d < L; d++) open_node(s[d]);
        if (skip.size() > (size_t)kTrieMaxNodes) return;   // too large: the per-token walk is used
        n_end[path.back()]++;
        dtok.push_back(t);
        prev = s;
        prev_len = L;
    }
    while (!path.empty()) close_node();
    const uint32_t N = (uint32_t)skip.size();
    // parents, branching heights and the classes below each node (children
    // have larger ids than their parent: one reverse pass)
    std::vector<uint32_t> parent(N, 0), bh(N, 0);
    std::vector<uint64_t> sub(N, 0);
    const bool subs = h->K <= 64;
    for (uint32_t n = N; n-- > 0;) {
        uint32_t m = 0, k = 0;
        for (uint32_t c = n + 1; c < skip[n]; c = skip[c]) {
            k++;
            parent[c] = n;
            m = std::max(m, bh[c]);
            if (subs) sub[n] |= (1ull << ncls[c]) | sub[c];
        }
        bh[n] = m + (k >= 2 ? 1u : 0u);
    }
    // upper nodes (an ancestor of an upper node is upper: subtree size and
    // branching height only grow towards the root), their paths, and the
    // units: the subtrees hanging off upper nodes
    std::vector<int32_t> uidx(N, -1);
    std::vector<uint4> upper;
    std::vector<uint8_t> upath;
    std::vector<uint2> unit;
    for (uint32_t n = 0; n < N;) {
        const bool up = n == 0 || skip[n] - n > (uint32_t)kTrieTile || bh[n] > (uint32_t)kTrieBranch;
        if (up) {
            uidx[n] = (int32_t)upper.size();
            const uint32_t off = (uint32_t)upath.size();
            uint32_t plen = 0;
            if (n != 0) {
                const uint4 pu = upper[(size_t)uidx[parent[n]]];
                upath.insert(upath.end(), upath.begin() + pu.y, upath.begin() + pu.y + pu.z);
                upath.push_back(ncls[n]);
                plen = pu.z + 1;
            }
            upper.push_back(make_uint4(n, off, plen, 0u));
            n++;
        } else {
            unit.push_back(make_uint2(n, (uint32_t)uidx[parent[n]]));
            n = skip[n];
        }
    }
    std::vector<uint4> node((size_t)N * 2);
    for (uint32_t n = 0; n < N; n++) {
        node[2 * (size_t)n] = make_uint4(skip[n] | ((uint32_t)ncls[n] << 24), tok_lo[n], n_end[n], tok_hi[n]);
        node[2 * (size_t)n + 1] = make_uint4((uint32_t)sub[n], (uint32_t)(sub[n] >> 32), 0u, 0u);
    }
    // Chains: inside a unit, a node with one child and no token ending at it
    // is walked together with that child.  The walk's records are the chains'
    // first nodes (heads); a record covers `len` nodes (at most 255), its
    // classes are those nodes' classes, and its tokens and classes-below are
    // those of its last node.  Upper nodes stay records of their own.
    std::vector<uint32_t> nchild(N, 0);
    for (uint32_t n = 1; n < N; n++) nchild[parent[n]]++;
    std::vector<uint8_t> head(N, 1);
    std::vector<uint32_t> clen(N, 1);   // a head's chain length
    for (const uint2& u : unit) {
        uint32_t cur = u.x;
        for (uint32_t n = u.x + 1; n < skip[u.x]; n++) {
            const uint32_t pp = parent[n];
            if (nchild[pp] == 1 && n_end[pp] == 0 && pp + 1 == n && clen[cur] < 255 &&
                cur + clen[cur] == n) {
                head[n] = 0;
                clen[cur]++;
            } else {
                cur = n;
            }
        }
    }
    std::vector<uint32_t> hc((size_t)N + 1, 0);   // heads before each node
    for (uint32_t n = 0; n < N; n++) hc[n + 1] = hc[n] + head[n];
    std::vector<uint4> cnode((size_t)hc[N] * 2);
    for (uint32_t n = 0; n < N; n++) {
        if (!head[n]) continue;
        const uint32_t b = n + clen[n] - 1;   // the chain's last node
        const size_t c = hc[n];
        cnode[2 * c] = make_uint4(hc[skip[n]], n, clen[n], tok_lo[n]);
        cnode[2 * c + 1] = make_uint4(n_end[b], (uint32_t)sub[b], (uint32_t)(sub[b] >> 32), 0u);
    }
    h->t_cnode.swap(cnode);
    h->t_hc.swap(hc);
    h->t_ncls.swap(ncls);
    h->t_node.swap(node);
    h->t_dtok.swap(dtok);
    h->t_upper.swap(upper);
    h->t_upath.swap(upath);
    h->t_unit.swap(unit);
    h->t_nodes = (int32_t)N;
    h->trie_built = true;
}

// Cuts the units into per-CTA batches that fit in the tile kernel's shared
// memory next to the transition table, for a grid of one CTA per SM.  Units
// are weighed by their estimated walk cost, cut in preorder into kTrieInterleave
// chunks per CTA of equal weight, and CTA c takes chunks c, c + grid, ...; a
// batch holds some of one CTA's units (staged as node, record and token ranges
// one after the other, costliest units first), the upper nodes they hang off
// (slots), and the upper nodes whose tokens it sets (emitting slots: each upper
// node with tokens is set by the batch of the first unit after it in preorder).
// Chooses the table placement: in shared memory when that leaves room for
// batches, else through L1/L2.  false: some unit alone does not fit (the
// per-token walk is used).
bool cut_batches(domino_ctx* h) {
    const int smem = h->env.max_smem_optin > 0 ? h->env.max_smem_optin : 232448;
    const int grid = h->env.num_sms > 0 ? h->env.num_sms : 1;
    StepView v = make_view(h);
    const bool self = !h->self_mask.empty();
    const std::vector<uint2>& unit = h->t_unit;
    const std::vector<uint4>& node = h->t_node;
    const std::vector<uint4>& upper = h->t_upper;
    auto skip_of = [&](uint32_t n) { return node[2 * (size_t)n].x & 0xFFFFFFu; };
    // fixed shared memory with an empty batch, per table placement
    TrieView tv0{};
    const int fixed = trie_tile_smem_bytes(v, tv0, h->stack, 0) + 1024;
    constexpr int kMinBatch = 24 * 1024;
    int mode = kDenseGlobal;
    int64_t table = 0;
    const int modes[2] = {kDenseSmem, h->sp_words == 2 ? kSparse32Smem : kSparse64Smem};
    for (int m : modes) {
        if (m != kDenseSmem && h->sp_nnz == 0) continue;
        const int64_t t = table_smem_bytes(v, h->stack, m);
        if ((int64_t)smem - fixed - t >= kMinBatch) {
            mode = m;
            table = t;
            break;
        }
    }
    // A unit costs about the transitions its walk takes, which depend on the
    // rows.  For a DFA they are counted here by walking the tree from up to
    // 1024 states spread evenly over the automaton (the visits inside each
    // unit); the CTAs' shares are balanced on those counts plus the units'
    // node counts.  Pushdown automata are balanced on node counts.
    std::vector<int64_t> unit_nodes(unit.size());
    for (size_t u = 0; u < unit.size(); u++) unit_nodes[u] = skip_of(unit[u].x) - unit[u].x;
    if (!h->stack && !h->t16.empty() && h->Q > 1 && !unit.empty()) {
        const int32_t Q = h->Q, K = h->K;
        const uint32_t N = skip_of(0);
        std::vector<int32_t> unit_of(N, -1);
        for (size_t u = 0; u < unit.size(); u++)
            for (uint32_t n = unit[u].x; n < skip_of(unit[u].x); n++) unit_of[n] = (int32_t)u;
        std::vector<int64_t> visits(unit.size(), 0);
        struct Frame {
            uint32_t next, end, s;
        };
        std::vector<Frame> stk;
        const int32_t stride = std::max<int32_t>(1, (Q - 1) / 1024);
        for (int32_t q = 1; q < Q; q += stride) {
            uint32_t n = 1, end = N, s = (uint32_t)q;
            stk.clear();
            for (;;) {
                if (n >= end) {
                    if (stk.empty()) break;
                    const Frame f = stk.back();
                    stk.pop_back();
                    n = f.next, end = f.end, s = f.s;
                    continue;
                }
                const uint32_t x = node[2 * (size_t)n].x, sk = x & 0xFFFFFFu;
                const uint32_t s2 = h->t16[(size_t)s * K + (x >> 24)];
                if (unit_of[n] >= 0) visits[(size_t)unit_of[n]]++;
                if (s2 != 0 && sk > n + 1) {
                    stk.push_back({sk, end, s});
                    n = n + 1, end = sk, s = s2;
                } else {
                    n = sk;
                }
            }
        }
        for (size_t u = 0; u < unit.size(); u++) unit_nodes[u] += visits[u];
    }
    int64_t total = 0;
    for (size_t u = 0; u < unit.size(); u++) total += unit_nodes[u];
    const int per_rec = 16 + (self ? 8 : 0);   // a staged walk record (and its classes below)
    const std::vector<uint32_t>& hc = h->t_hc;
    if (unit.empty()) return false;
    // the upper nodes whose tokens a unit's batch sets: those with tokens
    // between the previous unit's root and its own (trailing ones: the last)
    std::vector<std::vector<uint32_t>> emit_at(unit.size());
    {
        size_t ui = 0;
        for (size_t u = 0; u < upper.size(); u++) {
            if (node[2 * (size_t)upper[u].x].z == 0) continue;
            while (ui < unit.size() && unit[ui].x < upper[u].x) ui++;
            emit_at[std::min(ui, unit.size() - 1)].push_back((uint32_t)u);
        }
    }
    // The units in preorder are cut into grid x kTrieInterleave chunks of
    // equal cost; CTA c takes chunks c, c + grid, ...  The rows live at a
    // unit vary from one batch of rows to the next, and nearby units share
    // their upper nodes, so a CTA's share drawn from several places of the
    // tree varies less than one run of it.
    const int nchunk = grid * kTrieInterleave;
    std::vector<size_t> cbeg((size_t)nchunk + 1, unit.size());
    {
        int64_t done = 0;
        size_t u = 0;
        for (int j = 0; j < nchunk; j++) {
            cbeg[(size_t)j] = u;
            const int64_t goal = total * (j + 1) / nchunk;
            while (u < unit.size() && (done < goal || j == nchunk - 1)) done += unit_nodes[u++];
        }
    }
    for (int64_t budget = (int64_t)smem - fixed - table; budget >= 4096; budget = budget * 9 / 10) {
        std::vector<uint4> batch, slot, range;
        std::vector<uint2> bunit;
        std::vector<int64_t> bweight;   // the estimated cost of each bunit entry
        std::vector<int32_t> cta((size_t)grid + 1, 0);
        int32_t mx_nodes = 0, mx_cls = 0, mx_toks = 0, mx_units = 0, mx_slots = 0, mx_path = 0;
        bool ok = true;
        for (int c = 0; c < grid && ok; c++) {
            cta[(size_t)c] = (int32_t)(batch.size() / 2);
            std::vector<std::pair<size_t, size_t>> runs;   // this CTA's unit runs, in preorder
            for (int k = 0; k < kTrieInterleave; k++) {
                const size_t j = (size_t)c + (size_t)k * grid;
                if (cbeg[j] < cbeg[j + 1]) runs.emplace_back(cbeg[j], cbeg[j + 1]);
            }
            size_t ri = 0, u = runs.empty() ? 0 : runs[0].first;
            while (ri < runs.size() && ok) {
                // one batch: units of this CTA's runs from u on, staged as node
                // and token ranges one after the other
                const size_t slot0 = slot.size(), unit0 = bunit.size(), range0 = range.size();
                std::vector<std::pair<uint32_t, uint32_t>> slots;   // (upper index, slot)
                auto slot_of = [&](uint32_t ui, bool emit) -> int {
                    const uint32_t n = upper[ui].x;
                    for (auto& p : slots)
                        if (p.first == ui) {
                            if (emit) slot[slot0 + p.second].z = node[2 * (size_t)n].z;
                            return (int)p.second;
                        }
                    if ((int)slots.size() >= kTrieMaxSlots) return -1;
                    slot.push_back(make_uint4(ui, node[2 * (size_t)n].y, emit ? node[2 * (size_t)n].z : 0u, 0u));
                    slots.emplace_back(ui, (uint32_t)slots.size());
                    mx_path = std::max<int32_t>(mx_path, (int32_t)upper[ui].z);
                    return (int)slots.size() - 1;
                };
                int64_t recs_b = 0, cls_b = 0, toks_b = 0;   // staged by the closed ranges
                bool open = false;
                uint32_t rn0 = 0, rn1 = 0, rt0 = 0, rt1 = 0;   // the open range (nodes, tokens)
                auto close_range = [&]() {
                    if (!open) return;
                    range.push_back(make_uint4(hc[rn0], hc[rn1], rt0, rt1));
                    range.push_back(make_uint4(rn0, rn1, 0u, 0u));
                    recs_b += hc[rn1] - hc[rn0];
                    cls_b += rn1 - rn0;
                    toks_b += rt1 - rt0;
                    open = false;
                };
                size_t added = 0;
                while (ri < runs.size()) {
                    if (u >= runs[ri].second) {   // the run is done: its range closes
                        close_range();
                        if (++ri < runs.size()) u = runs[ri].first;
                        continue;
                    }
                    const size_t keep_slots = slot.size();
                    const auto keep_list = slots;
                    std::vector<uint32_t> keep_z;
                    for (size_t k = slot0; k < slot.size(); k++) keep_z.push_back(slot[k].z);
                    bool fit = true;
                    for (uint32_t e : emit_at[u])
                        if (fit) fit = slot_of(e, true) >= 0;
                    const int sl = fit ? slot_of(unit[u].y, false) : -1;
                    fit = sl >= 0;
                    const uint32_t n0 = open ? rn0 : unit[u].x, t0 = open ? rt0 : node[2 * (size_t)unit[u].x].y;
                    const uint32_t n1 = skip_of(unit[u].x), t1 = node[2 * (size_t)unit[u].x].w;
                    const int64_t recs_all = recs_b + (hc[n1] - hc[n0]), cls_all = cls_b + (n1 - n0);
                    const int64_t toks_all = toks_b + (t1 - t0);
                    if (fit)
                        fit = recs_all <= 0xFFFF && toks_all <= 0xFFFF &&
                              recs_all * per_rec + ((cls_all + 15) & ~15) + toks_all * 4 +
                                      (int64_t)(bunit.size() - unit0 + 1) * 4 + (int64_t)slots.size() * (16 + 64) <=
                                  budget;
                    if (!fit) {   // undo this unit's slots; the batch ends before it
                        slot.resize(keep_slots);
                        slots = keep_list;
                        for (size_t k = slot0; k < slot.size(); k++) slot[k].z = keep_z[k - slot0];
                        if (added == 0) ok = false;   // a unit alone does not fit
                        break;
                    }
                    bunit.push_back(make_uint2((uint32_t)(recs_b + (hc[unit[u].x] - hc[n0])), (uint32_t)sl));
                    bweight.push_back(unit_nodes[u]);
                    if (!open) {
                        rn0 = n0;
                        rt0 = t0;
                        open = true;
                    }
                    rn1 = n1;
                    rt1 = t1;
                    added++;
                    u++;
                }
                if (!ok) break;
                close_range();
                {   // the costliest units first: the warps' last claims are short ones
                    std::vector<size_t> ord(bunit.size() - unit0);
                    for (size_t k = 0; k < ord.size(); k++) ord[k] = unit0 + k;
                    std::stable_sort(ord.begin(), ord.end(),
                                     [&](size_t x, size_t y) { return bweight[x] > bweight[y]; });
                    std::vector<uint2> su;
                    std::vector<int64_t> sw;
                    for (size_t k : ord) {
                        su.push_back(bunit[k]);
                        sw.push_back(bweight[k]);
                    }
                    std::copy(su.begin(), su.end(), bunit.begin() + (ptrdiff_t)unit0);
                    std::copy(sw.begin(), sw.end(), bweight.begin() + (ptrdiff_t)unit0);
                }
                batch.push_back(make_uint4((uint32_t)unit0, (uint32_t)bunit.size(), (uint32_t)(range0 / 2),
                                           (uint32_t)(range.size() / 2)));
                batch.push_back(make_uint4((uint32_t)slot0, (uint32_t)slot.size(), (uint32_t)recs_b,
                                           (uint32_t)toks_b));
                mx_nodes = std::max<int32_t>(mx_nodes, (int32_t)recs_b);
                mx_cls = std::max<int32_t>(mx_cls, (int32_t)cls_b);
                mx_toks = std::max<int32_t>(mx_toks, (int32_t)toks_b);
                mx_units = std::max<int32_t>(mx_units, (int32_t)(bunit.size() - unit0));
                mx_slots = std::max<int32_t>(mx_slots, (int32_t)(slot.size() - slot0));
            }
        }
        if (!ok) continue;
        cta[(size_t)grid] = (int32_t)(batch.size() / 2);
        TrieView tv{};
        tv.max_nodes = mx_nodes;
        tv.max_cls = mx_cls;
        tv.max_toks = mx_toks;
        tv.max_units = mx_units;
        tv.max_slots = mx_slots;
        tv.max_path = mx_path;
        if (trie_tile_smem_bytes(v, tv, h->stack, (int)table) > smem) continue;   // the maxima together: cut tighter
        h->t_batch.swap(batch);
        h->t_range.swap(range);
        h->t_slot.swap(slot);
        h->t_bunit.swap(bunit);
        h->t_cta.swap(cta);
        h->t_grid = grid;
        h->t_max_nodes = mx_nodes;
        h->t_max_cls = mx_cls;
        h->t_max_toks = mx_toks;
        h->t_max_units = mx_units;
        h->t_max_slots = mx_slots;
        h->t_max_path = mx_path;
        h->t_mode = mode;
        return true;
    }
    return false;
}

// The prefix tree and its batches on the device.
int build_trie(domino_ctx* h) {
    build_trie_host(h);
    if (!h->trie_built || !cut_batches(h)) return DOMINO_OK;
    int rc;
    auto up = [&](DevBuf& b, const void* p, size_t n) { return dev_upload(b, p, std::max<size_t>(16, n)); };
    if ((rc = up(h->d_tnode, h->t_cnode.data(), h->t_cnode.size() * sizeof(uint4)))) return rc;
    if ((rc = up(h->d_tncls, h->t_ncls.data(), h->t_ncls.size()))) return rc;
    if ((rc = up(h->d_tdtok, h->t_dtok.data(), h->t_dtok.size() * 4))) return rc;
    if ((rc = up(h->d_tupper, h->t_upper.data(), h->t_upper.size() * sizeof(uint4)))) return rc;
    if ((rc = up(h->d_tupath, h->t_upath.data(), h->t_upath.size()))) return rc;
    if ((rc = up(h->d_tbatch, h->t_batch.data(), h->t_batch.size() * sizeof(uint4)))) return rc;
    if ((rc = up(h->d_trange, h->t_range.data(), h->t_range.size() * sizeof(uint4)))) return rc;
    if ((rc = up(h->d_tslot, h->t_slot.data(), h->t_slot.size() * sizeof(uint4)))) return rc;
    if ((rc = up(h->d_tunit, h->t_bunit.data(), h->t_bunit.size() * sizeof(uint2)))) return rc;
    if ((rc = up(h->d_tcta, h->t_cta.data(), h->t_cta.size() * 4))) return rc;
    if ((rc = dev_reserve(h->d_trow, std::max<size_t>(1, h->t_batch.size() / 2) * 4))) return rc;
    h->trie_ready = true;
    return DOMINO_OK;
}

// Byte-class strings of every token, the window sort and the slot arrays.
int build_arena(domino_ctx* h) {
    h->arena_ready = false;
    if (!h->vocab_loaded || !h->auto_loaded) return DOMINO_OK;
    const int32_t V = h->V;
    const int32_t nw = (V + kWin - 1) / kWin;
    const int64_t n_slots = (int64_t)nw * kWin;
    std::vector<uint8_t> cls(h->tok_bytes.size());
    for (size_t i = 0; i < cls.size(); i++) cls[i] = h->byte_class[h->tok_bytes[i]];
    auto tlen = [&](int32_t t) -> int32_t {
        return t == h->eos_id ? 0 : (int32_t)(h->tok_off[t + 1] - h->tok_off[t]);
    };
    // window order: empty tokens first, then by first class; inside a first-class
    // group longer tokens first (a warp's lanes then walk similar lengths), then
    // by class string (shared prefixes take the same transitions)
    auto less = [&](int32_t a, int32_t b) {
        int32_t la = tlen(a), lb = tlen(b);
        if ((la == 0) != (lb == 0)) return la == 0;
        if (la == 0) return a < b;
        const uint8_t* ca = cls.data() + h->tok_off[a];
        const uint8_t* cb = cls.data() + h->tok_off[b];
        if (ca[0] != cb[0]) return ca[0] < cb[0];
        if (la != lb) return la > lb;
        int c = std::memcmp(ca, cb, (size_t)la);
        if (c != 0) return c < 0;
        return a < b;
    };
    const int K = h->K;
    std::vector<uint8_t> head((size_t)n_slots * kInlineBytes, 0);
    const bool self = !h->self_mask.empty();
    std::vector<uint64_t> tok_cls(self ? (size_t)n_slots : 0, 0);   // classes of bytes 1.. of each slot
    std::vector<uint32_t> info((size_t)n_slots, 0);
    std::vector<int32_t> tail_off((size_t)n_slots, 0), pos_of((size_t)V, 0);
    std::vector<uint16_t> gstart((size_t)(K + 1), 0);
    std::vector<uint16_t> cls_start((size_t)nw * (size_t)(h->K + 1), 0);   // [window][class]: first slot
    std::vector<int16_t> eos_slot((size_t)nw, -1);
    std::vector<uint8_t> tail;
    std::vector<int32_t> ids;
    for (int32_t w = 0; w < nw; w++) {
        int32_t lo = w * kWin, hi = std::min(V, lo + kWin);
        ids.resize((size_t)(hi - lo));
        std::iota(ids.begin(), ids.end(), lo);
        std::sort(ids.begin(), ids.end(), less);
        uint16_t* gs = gstart.data();
        int c_next = 0;   // first class whose group start is still unset
        for (int32_t j = 0; j < hi - lo; j++) {
            int32_t t = ids[(size_t)j];
            int64_t p = (int64_t)lo + j;
            int32_t L = tlen(t);
            info[(size_t)p] = (uint32_t)(t - lo) | kInfoValid | ((uint32_t)L << 16);
            pos_of[(size_t)t] = (int32_t)p;
            if (t == h->eos_id) eos_slot[(size_t)w] = (int16_t)j;
            const uint8_t* c = cls.data() + h->tok_off[t];
            if (L > 0) {
                while (c_next <= c[0]) gs[c_next++] = (uint16_t)j;   // groups by first class
            }
            std::memcpy(head.data() + p * kInlineBytes, c, (size_t)std::min(L, kInlineBytes));
            if (self)
                for (int32_t i = 1; i < L; i++) tok_cls[(size_t)p] |= 1ull << c[i];
            if (L > kInlineBytes) {
                tail_off[(size_t)p] = (int32_t)tail.size();
                tail.insert(tail.end(), c + kInlineBytes, c + L);
            }
        }
        while (c_next <= K) gs[c_next++] = (uint16_t)(hi - lo);
        // the slots of first class c are [gs[c], gs[c + 1]) of the window
        std::copy(gs, gs + K + 1, cls_start.begin() + (ptrdiff_t)((size_t)w * (K + 1)));
    }
    if (tail.size() > (size_t)INT32_MAX) return DOMINO_E_UNSUPPORTED;
    int rc;
    if ((rc = dev_upload(h->d_head, head.data(), head.size()))) return rc;
    if ((rc = dev_upload(h->d_info, info.data(), info.size() * 4))) return rc;
    if ((rc = dev_upload(h->d_tail_off, tail_off.data(), tail_off.size() * 4))) return rc;
    if ((rc = dev_upload(h->d_tail, tail.data(), tail.size()))) return rc;
    if ((rc = dev_upload(h->d_pos_of, pos_of.data(), pos_of.size() * 4))) return rc;
    if ((rc = dev_upload(h->d_cls_start, cls_start.data(), cls_start.size() * 2))) return rc;
    if (self) {
        if ((rc = dev_upload(h->d_tok_cls, tok_cls.data(), tok_cls.size() * 8))) return rc;
    } else {
        dev_free(h->d_tok_cls);
    }
    if ((rc = dev_upload(h->d_eos_slot, eos_slot.data(), eos_slot.size() * 2))) return rc;
    h->n_windows = nw;
    if ((rc = build_trie(h))) return rc;
    h->arena_ready = true;
    return DOMINO_OK;
}

StepView make_view(domino_ctx* h) {
    StepView v{};
    v.head = (const uint4*)h->d_head.p;
    v.info = (const uint32_t*)h->d_info.p;
    v.tail_off = (const int32_t*)h->d_tail_off.p;
    v.tail = (const uint8_t*)h->d_tail.p;
    v.pos_of = (const int32_t*)h->d_pos_of.p;
    v.cls_start = (const uint16_t*)h->d_cls_start.p;
    v.eos_slot = (const int16_t*)h->d_eos_slot.p;
    v.V = h->V;
    v.W = h->W;
    v.n_windows = h->n_windows;
    v.eos_id = h->eos_id;
    const char* dense = (const char*)h->d_dense.p;
    v.t16 = h->stack ? nullptr : (const uint16_t*)dense;
    v.t32 = h->stack ? (const uint32_t*)dense : nullptr;
    v.ret = dense ? (const uint16_t*)(dense + h->dense_ret_off) : nullptr;
    v.sp_info = (const uint32_t*)h->d_sparse.p;
    v.sp_tgt = h->d_sparse.p ? (const void*)((const char*)h->d_sparse.p + h->sp_tgt_off) : nullptr;
    v.accept_bits = (const uint32_t*)h->d_accept.p;
    v.self_mask = h->self_mask.empty() ? nullptr : (const unsigned long long*)h->d_self.p;
    v.tok_cls = h->self_mask.empty() ? nullptr : (const unsigned long long*)h->d_tok_cls.p;
    v.Q = h->Q;
    v.K = h->K;
    v.start = h->start;
    v.max_depth = h->max_depth;
    v.n_ret = (int32_t)(h->ret.size() / 4);
    v.sp_nnz = h->sp_nnz;
    v.err = (uint32_t*)h->d_err.p;
    return v;
}

// Table placement for the step kernel: dense in shared memory if it fits, else
// the sparse live-class form, else dense through L1/L2.
int choose_mode(const domino_ctx* h, const StepView& v, bool next) {
    if (h->env.max_smem_optin <= 0) return kDenseGlobal;
    const int64_t avail = (int64_t)h->env.max_smem_optin - step_fixed_smem_bytes(v, next) - 1024;
    if (table_smem_bytes(v, h->stack, kDenseSmem) <= avail) return kDenseSmem;
    if (h->sp_nnz > 0) {
        const int mode = h->sp_words == 2 ? kSparse32Smem : kSparse64Smem;
        if (table_smem_bytes(v, h->stack, mode) <= avail) return mode;
    }
    return kDenseGlobal;
}

TrieView make_trie_view(const domino_ctx* h) {
    TrieView tv{};
    tv.node = (const uint4*)h->d_tnode.p;
    tv.ncls = (const uint8_t*)h->d_tncls.p;
    tv.dtok = (const int32_t*)h->d_tdtok.p;
    tv.upper = (const uint4*)h->d_tupper.p;
    tv.upath = (const uint8_t*)h->d_tupath.p;
    tv.batch = (const uint4*)h->d_tbatch.p;
    tv.range = (const uint4*)h->d_trange.p;
    tv.slot = (const uint4*)h->d_tslot.p;
    tv.unit = (const uint2*)h->d_tunit.p;
    tv.cta_batch = (const int32_t*)h->d_tcta.p;
    tv.n_nodes = h->t_nodes;
    tv.n_upper = (int32_t)h->t_upper.size();
    tv.grid = h->t_grid;
    tv.n_batches = (int32_t)(h->t_batch.size() / 2);
    tv.max_nodes = h->t_max_nodes;
    tv.max_cls = h->t_max_cls;
    tv.max_toks = h->t_max_toks;
    tv.max_units = h->t_max_units;
    tv.max_slots = h->t_max_slots;
    tv.max_path = h->t_max_path;
    return tv;
}

// The tree shares each prefix's transitions among the tokens below it and
// drops a subtree as soon as its prefix dies, so it wins when most prefixes
// die early (sparse masks).  States that loop on many classes (strings,
// numbers, whitespace: the self-loop mask) keep long prefixes alive and make
// rows dense; there the per-token walk, which skips a whole token whose later
// classes all loop on the state, is faster.
bool use_tree(const domino_ctx* h) {
    if (!h->trie_ready || h->walk_pref == 0) return false;
    return h->walk_pref == 1 || h->self_mask.empty();
}

int ready_for_compute(domino_ctx* h) {
    if (!h) return DOMINO_E_INVALID_ARG;
    if (is_host_only(h)) return DOMINO_E_NO_DEVICE;
    if (!h->vocab_loaded || !h->auto_loaded || !h->arena_ready) return DOMINO_E_NOT_LOADED;
    return DOMINO_OK;
}

int cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return DOMINO_OK;
    cudaGetLastError();
    return DOMINO_E_CUDA;
}

// An NVTX range named after each C ABI call that does work (a no-op unless a
// profiler is attached), so that a timeline shows the library's calls above
// the kernels they launch.
struct ApiRange {
    explicit ApiRange(const char* name) { nvtxRangePushA(name); }
    ~ApiRange() { nvtxRangePop(); }
    ApiRange(const ApiRange&) = delete;
    ApiRange& operator=(const ApiRange&) = delete;
};
#define DOMINO_API_RANGE() const ApiRange api_range_(__func__)

}  // namespace

extern "C" {

const char* domino_status_string(int s) {
    switch (s) {
        case DOMINO_OK: return "ok";
        case DOMINO_E_INVALID_ARG: return "invalid argument";
        case DOMINO_E_NOT_LOADED: return "vocabulary or automaton not loaded";
        case DOMINO_E_UNSUPPORTED: return "unsupported request";
        case DOMINO_E_OOM: return "out of memory";
        case DOMINO_E_CUDA: return "CUDA runtime error";
        case DOMINO_E_NO_DEVICE: return "host-only handle has no device";
        default: return "unknown status";
    }
}

int domino_create(domino_t* out, int32_t cuda_device) {
    if (!out) return DOMINO_E_INVALID_ARG;
    *out = nullptr;
    domino_ctx* h = new (std::nothrow) domino_ctx();
    if (!h) return DOMINO_E_OOM;
    h->device = cuda_device < 0 ? -1 : cuda_device;
    if (const char* w = std::getenv("DOMINO_WALK")) {
        if (std::strcmp(w, "token") == 0) h->walk_pref = 0;
        if (std::strcmp(w, "tree") == 0) h->walk_pref = 1;
    }
    if (h->device >= 0) {
        int n = 0;
        if (cudaGetDeviceCount(&n) != cudaSuccess || cuda_device >= n) {
            cudaGetLastError();
            delete h;
            return cuda_device >= n && n > 0 ? DOMINO_E_INVALID_ARG : DOMINO_E_CUDA;
        }
        if (cudaSetDevice(h->device) != cudaSuccess) {
            cudaGetLastError();
            delete h;
            return DOMINO_E_CUDA;
        }
        cudaDeviceGetAttribute(&h->env.num_sms, cudaDevAttrMultiProcessorCount, h->device);
        cudaDeviceGetAttribute(&h->env.max_smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, h->device);
        int rc = prepare_logits_kernels() == cudaSuccess ? DOMINO_OK : DOMINO_E_CUDA;
        if (!rc) rc = dev_reserve(h->d_err, 16);
        if (!rc) rc = dev_reserve(h->d_partials, sizeof(float4) * (size_t)kMaxLogitRows * kMaxSegments);
        if (!rc) rc = dev_reserve(h->d_counters, sizeof(uint32_t) * (size_t)kMaxLogitRows);
        if (!rc) rc = dev_reserve(h->d_lse_tmp, sizeof(float) * (size_t)kMaxLogitRows);
        if (!rc && (cudaMemset(h->d_err.p, 0, 16) != cudaSuccess ||
                    cudaMemset(h->d_counters.p, 0, sizeof(uint32_t) * (size_t)kMaxLogitRows) != cudaSuccess)) {
            cudaGetLastError();
            rc = DOMINO_E_CUDA;
        }
        if (rc) {
            domino_destroy(h);
            return rc;
        }
    }
    *out = h;
    return DOMINO_OK;
}

int domino_destroy(domino_t h) {
    if (!h) return DOMINO_OK;
    if (h->device >= 0) {
        DeviceGuard g(h->device);
        cudaDeviceSynchronize();
        DevBuf* all[] = {&h->d_head, &h->d_info, &h->d_tail_off, &h->d_tail, &h->d_pos_of, &h->d_cls_start,
                         &h->d_eos_slot, &h->d_dense, &h->d_sparse, &h->d_accept, &h->d_self, &h->d_tok_cls, &h->d_err, &h->d_fpart, &h->d_partials,
                         &h->d_counters, &h->d_lse_tmp, &h->s_logits, &h->s_mask, &h->s_io,
                         &h->o_prop, &h->o_rows, &h->o_count, &h->d_tnode, &h->d_tdtok, &h->d_tupper, &h->d_tupath, &h->d_tbatch, &h->d_tslot,
                         &h->d_tunit, &h->d_tcta, &h->d_trange, &h->d_tncls, &h->d_trow};
        for (auto* b : all) dev_free(*b);
        for (cudaEvent_t& e : h->ev_chunk)
            if (e) cudaEventDestroy(e);
        for (cudaEvent_t& e : h->ev_t)
            if (e) cudaEventDestroy(e);
        if (h->ev_cfg) cudaEventDestroy(h->ev_cfg);
        if (h->cp_stream) cudaStreamDestroy(h->cp_stream);
        if (h->h_io) cudaFreeHost(h->h_io);
        clear_host_graphs(h);
        cudaGetLastError();
    }
    delete h;
    return DOMINO_OK;
}

int domino_load_vocab(domino_t h, const uint8_t* bytes, const int64_t* offsets, int32_t n_tokens,
                      int32_t eos_id) {
    DOMINO_API_RANGE();
    if (h) clear_host_graphs(h);
    if (!h || !offsets || n_tokens < 1 || n_tokens > (1 << 24)) return DOMINO_E_INVALID_ARG;
    if (eos_id < -1 || eos_id >= n_tokens || offsets[0] != 0) return DOMINO_E_INVALID_ARG;
    int32_t max_len = 0;
    for (int32_t t = 0; t < n_tokens; t++) {
        int64_t L = offsets[t + 1] - offsets[t];
        if (L < 0 || L > 65535) return DOMINO_E_INVALID_ARG;
        if (t != eos_id) max_len = std::max<int32_t>(max_len, (int32_t)L);
    }
    if (offsets[n_tokens] > 0 && !bytes) return DOMINO_E_INVALID_ARG;
    DeviceGuard g(h->device);
    h->vocab_loaded = false;
    h->arena_ready = false;
    h->tok_off.assign(offsets, offsets + n_tokens + 1);
    if (bytes && offsets[n_tokens] > 0)
        h->tok_bytes.assign(bytes, bytes + offsets[n_tokens]);
    else
        h->tok_bytes.clear();
    h->V = n_tokens;
    h->W = (n_tokens + 31) / 32;
    h->eos_id = eos_id;
    h->max_len = max_len;
    h->vocab_loaded = true;
    if (is_host_only(h)) {
        build_trie_host(h);
        return DOMINO_OK;
    }
    return build_arena(h);
}

int domino_load_automaton(domino_t h, const int32_t* delta, int32_t n_states, const uint8_t* live,
                          const uint8_t* accepting, int32_t start_state, const domino_stack_rule* rules,
                          int32_t n_rules, int32_t max_depth) {
    DOMINO_API_RANGE();
    if (!h || !delta || !live || n_states < 1 || n_states > DOMINO_MAX_STATES) return DOMINO_E_INVALID_ARG;
    if (start_state < 0 || start_state >= n_states || max_depth < 0 || max_depth > DOMINO_MAX_DEPTH)
        return DOMINO_E_INVALID_ARG;
    if (n_rules < 0 || (n_rules > 0 && !rules)) return DOMINO_E_INVALID_ARG;
    const int64_t Q = n_states;
    for (int64_t i = 0; i < Q * 256; i++)
        if (delta[i] < 0 || delta[i] >= n_states) return DOMINO_E_INVALID_ARG;
    if (live[0]) return DOMINO_E_INVALID_ARG;
    for (int c = 0; c < 256; c++)
        if (delta[c] != 0) return DOMINO_E_INVALID_ARG;          // state 0 absorbing
    for (int64_t q = 0; q < Q; q++)
        if (accepting && accepting[q] && !live[q]) return DOMINO_E_INVALID_ARG;
    // rules: one per (state, byte); index -1 = none
    std::vector<int32_t> rule_at((size_t)(Q * 256), -1);
    for (int32_t r = 0; r < n_rules; r++) {
        const domino_stack_rule& R = rules[r];
        if (R.state <= 0 || R.state >= n_states || R.pad != 0 || R.sym > 1 ||
            (R.kind != DOMINO_RULE_PUSH && R.kind != DOMINO_RULE_POP))
            return DOMINO_E_INVALID_ARG;
        if (R.kind == DOMINO_RULE_POP) {
            for (int32_t t : {R.next_if_empty, R.next_if_top0, R.next_if_top1})
                if (t < 0 || t >= n_states) return DOMINO_E_INVALID_ARG;
        }
        int32_t& slot = rule_at[(size_t)R.state * 256 + R.byte];
        if (slot != -1) return DOMINO_E_INVALID_ARG;
        slot = r;
    }
    // closure: a non-live state only reaches non-live states (makes early exit exact)
    for (int64_t q = 0; q < Q; q++) {
        if (live[q]) continue;
        for (int c = 0; c < 256; c++) {
            int32_t r = rule_at[(size_t)q * 256 + c];
            if (r >= 0 && rules[r].kind == DOMINO_RULE_POP) {
                if (live[rules[r].next_if_empty] || live[rules[r].next_if_top0] || live[rules[r].next_if_top1])
                    return DOMINO_E_INVALID_ARG;
            } else if (live[delta[q * 256 + c]]) {
                return DOMINO_E_INVALID_ARG;
            }
        }
    }
    auto canon = [&](int32_t t) -> uint32_t { return live[t] ? (uint32_t)t : 0u; };
    // full entry for every (q, byte): dead-canonicalised, pop targets as deduplicated triples
    const bool stack = n_rules > 0;
    std::vector<uint32_t> col((size_t)(256 * Q));   // column-major: [byte][q]
    std::vector<uint16_t> ret;
    std::unordered_map<uint64_t, uint32_t> triple_id;
    for (int64_t q = 0; q < Q; q++) {
        for (int c = 0; c < 256; c++) {
            int32_t r = rule_at[(size_t)q * 256 + c];
            uint32_t e;
            if (r < 0) {
                e = canon(delta[q * 256 + c]);
            } else if (rules[r].kind == DOMINO_RULE_PUSH) {
                e = canon(delta[q * 256 + c]) | (1u << kKindShift) | ((uint32_t)rules[r].sym << kSymShift);
            } else {
                uint64_t key = ((uint64_t)canon(rules[r].next_if_empty) << 32) |
                               ((uint64_t)canon(rules[r].next_if_top0) << 16) | canon(rules[r].next_if_top1);
                auto it = triple_id.find(key);
                uint32_t id;
                if (it == triple_id.end()) {
                    id = (uint32_t)(ret.size() / 4);
                    if (id >= kMaxRetTriples) return DOMINO_E_UNSUPPORTED;
                    triple_id.emplace(key, id);
                    ret.push_back((uint16_t)canon(rules[r].next_if_empty));
                    ret.push_back((uint16_t)canon(rules[r].next_if_top0));
                    ret.push_back((uint16_t)canon(rules[r].next_if_top1));
                    ret.push_back(0);
                } else {
                    id = it->second;
                }
                e = (2u << kKindShift) | ((uint32_t)rules[r].sym << kSymShift) | (id << kRetShift);
            }
            col[(size_t)c * Q + q] = e;
        }
    }
    // byte classes: bytes whose columns are identical for every state
    uint8_t cls[256];
    int rep[256];
    int K = 0;
    std::unordered_map<uint64_t, std::vector<int>> by_hash;
    for (int c = 0; c < 256; c++) {
        const uint32_t* cc = col.data() + (size_t)c * Q;
        uint64_t hsh = 1469598103934665603ull;
        for (int64_t q = 0; q < Q; q++) hsh = (hsh ^ cc[q]) * 1099511628211ull;
        int found = -1;
        for (int k : by_hash[hsh]) {
            if (std::memcmp(cc, col.data() + (size_t)rep[k] * Q, sizeof(uint32_t) * (size_t)Q) == 0) {
                found = k;
                break;
            }
        }
        if (found < 0) {
            found = K++;
            rep[found] = c;
            by_hash[hsh].push_back(found);
        }
        cls[c] = (uint8_t)found;
    }
    DeviceGuard g(h->device);
    clear_host_graphs(h);
    h->auto_loaded = false;
    h->arena_ready = false;
    h->Q = n_states;
    h->K = K;
    h->start = start_state;
    h->max_depth = max_depth;
    h->n_rules = n_rules;
    h->stack = stack;
    std::memcpy(h->byte_class, cls, 256);
    h->t16.clear();
    h->t32.clear();
    if (stack) {
        h->t32.resize((size_t)(Q * K));
        for (int64_t q = 0; q < Q; q++)
            for (int k = 0; k < K; k++) h->t32[(size_t)(q * K + k)] = col[(size_t)rep[k] * Q + q];
    } else {
        h->t16.resize((size_t)(Q * K));
        for (int64_t q = 0; q < Q; q++)
            for (int k = 0; k < K; k++) h->t16[(size_t)(q * K + k)] = (uint16_t)col[(size_t)rep[k] * Q + q];
    }
    h->ret = ret;
    // Self loops: class k keeps state q (with no stack action).  A token whose
    // remaining classes all keep the row's state leaves it unchanged, so the
    // walk can skip it.  Used when some state loops on at least a quarter of
    // the classes: the string, number and whitespace states of real grammars.
    h->self_mask.clear();
    if (K <= 64) {
        std::vector<uint64_t> sm((size_t)Q, 0);
        bool wide = false;
        for (int64_t q = 1; q < Q; q++) {
            for (int k = 0; k < K; k++) {
                const uint32_t e = stack ? h->t32[(size_t)(q * K + k)] : h->t16[(size_t)(q * K + k)];
                if (e == (uint32_t)q) sm[(size_t)q] |= 1ull << k;   // next state q, kind 0 (no push or pop)
            }
            wide = wide || 4 * __builtin_popcountll(sm[(size_t)q]) >= K;
        }
        if (wide) h->self_mask.swap(sm);
    }
    h->accept_bits.assign((size_t)((Q + 31) / 32), 0u);
    if (accepting)
        for (int64_t q = 0; q < Q; q++)
            if (accepting[q]) h->accept_bits[(size_t)(q / 32)] |= 1u << (q % 32);
    h->auto_loaded = true;
    // dense image: [Q][K] entries | pop targets, each part 16-byte aligned
    const size_t esz = stack ? 4 : 2;
    auto a16 = [](size_t x) { return (x + 15) / 16 * 16; };
    const size_t tab_bytes = (size_t)(Q * K) * esz;
    h->dense_ret_off = (int64_t)a16(tab_bytes);
    std::vector<uint8_t> dense_img(a16(tab_bytes) + a16(h->ret.size() * 2), 0);
    std::memcpy(dense_img.data(), stack ? (const void*)h->t32.data() : (const void*)h->t16.data(), tab_bytes);
    if (!h->ret.empty()) std::memcpy(dense_img.data() + h->dense_ret_off, h->ret.data(), h->ret.size() * 2);
    // sparse image (K <= 64): per state {live-class mask, base} | live entries | pop targets
    h->sp_nnz = 0;
    h->sp_words = 0;
    std::vector<uint8_t> sparse_img;
    if (K <= 64) {
        const int words = K <= 32 ? 2 : 4;
        std::vector<uint32_t> rinfo((size_t)(Q * words), 0);
        std::vector<uint32_t> tgt;
        for (int64_t q = 0; q < Q; q++) {
            uint64_t m = 0;
            uint32_t base = (uint32_t)tgt.size();
            for (int k = 0; k < K; k++) {
                uint32_t e = stack ? h->t32[(size_t)(q * K + k)] : h->t16[(size_t)(q * K + k)];
                if (e) {
                    m |= 1ull << k;
                    tgt.push_back(e);
                }
            }
            if (words == 2) {
                rinfo[(size_t)(q * 2)] = (uint32_t)m;
                rinfo[(size_t)(q * 2 + 1)] = base;
            } else {
                rinfo[(size_t)(q * 4)] = (uint32_t)m;
                rinfo[(size_t)(q * 4 + 1)] = (uint32_t)(m >> 32);
                rinfo[(size_t)(q * 4 + 2)] = base;
            }
        }
        if (!tgt.empty() && tgt.size() < (size_t)INT32_MAX) {
            h->sp_nnz = (int32_t)tgt.size();
            h->sp_words = words;
            h->sp_tgt_off = (int64_t)a16(rinfo.size() * 4);
            h->sp_ret_off = h->sp_tgt_off + (int64_t)a16(tgt.size() * esz);
            sparse_img.assign((size_t)h->sp_ret_off + a16(h->ret.size() * 2), 0);
            std::memcpy(sparse_img.data(), rinfo.data(), rinfo.size() * 4);
            uint8_t* tp = sparse_img.data() + h->sp_tgt_off;
            for (size_t i = 0; i < tgt.size(); i++) {
                if (stack) {
                    std::memcpy(tp + i * 4, &tgt[i], 4);
                } else {
                    uint16_t e16 = (uint16_t)tgt[i];
                    std::memcpy(tp + i * 2, &e16, 2);
                }
            }
            if (!h->ret.empty()) std::memcpy(sparse_img.data() + h->sp_ret_off, h->ret.data(), h->ret.size() * 2);
        }
    }
    if (is_host_only(h)) {
        build_trie_host(h);
        return DOMINO_OK;
    }
    int rc;
    if ((rc = dev_upload(h->d_dense, dense_img.data(), dense_img.size()))) return rc;
    if (!sparse_img.empty()) {
        if ((rc = dev_upload(h->d_sparse, sparse_img.data(), sparse_img.size()))) return rc;
    } else {
        dev_free(h->d_sparse);
    }
    if ((rc = dev_upload(h->d_accept, h->accept_bits.data(), h->accept_bits.size() * 4))) return rc;
    if (!h->self_mask.empty()) {
        if ((rc = dev_upload(h->d_self, h->self_mask.data(), h->self_mask.size() * 8))) return rc;
    } else {
        dev_free(h->d_self);
    }
    return build_arena(h);
}

int domino_get_info(domino_t h, domino_info* out) {
    if (!h || !out) return DOMINO_E_INVALID_ARG;
    std::memset(out, 0, sizeof(*out));
    out->n_tokens = h->V;
    out->n_words = h->W;
    out->eos_id = h->eos_id;
    out->max_token_len = h->max_len;
    out->n_states = h->Q;
    out->n_classes = h->K;
    out->start_state = h->start;
    out->max_depth = h->max_depth;
    out->n_rules = h->n_rules;
    out->has_stack = h->stack ? 1 : 0;
    out->device = h->device;
    if (h->auto_loaded && h->device >= 0) {
        StepView v = make_view(h);
        out->table_in_smem = choose_mode(h, v, false) != kDenseGlobal ? 1 : 0;
    }
    out->device_bytes = dev_bytes(h);
    out->walk_tree = use_tree(h) ? 1 : 0;
    out->tree_units = h->trie_ready ? (int32_t)h->t_bunit.size() : 0;
    return DOMINO_OK;
}

int domino_get_byte_classes(domino_t h, uint8_t* classes_out) {
    if (!h || !classes_out) return DOMINO_E_INVALID_ARG;
    if (!h->auto_loaded) return DOMINO_E_NOT_LOADED;
    std::memcpy(classes_out, h->byte_class, 256);
    return DOMINO_OK;
}

int domino_get_prefix_tree(domino_t h, uint32_t* nodes_out, int64_t nodes_cap, int32_t* tokens_out,
                           int64_t tokens_cap, uint32_t* upper_out, int64_t upper_cap, uint32_t* units_out,
                           int64_t units_cap, int64_t* sizes_out) {
    if (!h || !sizes_out || nodes_cap < 0 || tokens_cap < 0 || upper_cap < 0 || units_cap < 0)
        return DOMINO_E_INVALID_ARG;
    if (!h->vocab_loaded || !h->auto_loaded) return DOMINO_E_NOT_LOADED;
    if (!h->trie_built) return DOMINO_E_UNSUPPORTED;
    const int64_t nu = (int64_t)h->t_upper.size(), nn = (int64_t)h->t_unit.size();
    sizes_out[0] = h->t_nodes;
    sizes_out[1] = (int64_t)h->t_dtok.size();
    sizes_out[2] = nu;
    sizes_out[3] = nn;
    if (nodes_out)
        std::memcpy(nodes_out, h->t_node.data(), (size_t)std::min<int64_t>(nodes_cap, h->t_nodes) * 2 * sizeof(uint4));
    if (tokens_out)
        std::memcpy(tokens_out, h->t_dtok.data(), (size_t)std::min<int64_t>(tokens_cap, (int64_t)h->t_dtok.size()) * 4);
    for (int64_t i = 0; upper_out && i < std::min(upper_cap, nu); i++) {
        upper_out[2 * i] = h->t_upper[(size_t)i].x;
        upper_out[2 * i + 1] = h->t_upper[(size_t)i].z;
    }
    for (int64_t i = 0; units_out && i < std::min(units_cap, nn); i++) {
        units_out[2 * i] = h->t_unit[(size_t)i].x;
        units_out[2 * i + 1] = h->t_unit[(size_t)i].y;
    }
    return DOMINO_OK;
}

int domino_step_mask(domino_t h, const int32_t* states_dev, const uint64_t* stacks_dev, int32_t batch,
                     uint32_t* mask_dev, int32_t* next_dev, void* stream) {
    DOMINO_API_RANGE();
    int rc = ready_for_compute(h);
    if (rc) return rc;
    if (batch < 0 || (batch > 0 && (!states_dev || !mask_dev))) return DOMINO_E_INVALID_ARG;
    if (batch == 0) return DOMINO_OK;
    DeviceGuard g(h->device);
    StepView v = make_view(h);
    if (use_tree(h)) {
        return cuda_status(launch_trie_step(v, make_trie_view(h), h->env, h->stack, h->t_mode, states_dev, stacks_dev,
                                            batch, false, mask_dev, next_dev, (cudaStream_t)stream));
    }
    const int mode = choose_mode(h, v, next_dev != nullptr);
    return cuda_status(launch_step_mask(v, h->env, h->stack, mode, states_dev, stacks_dev, batch, false, mask_dev,
                                        next_dev, (cudaStream_t)stream));
}

int domino_precompute_table(domino_t h, int32_t* next_dev, uint32_t* mask_dev, void* stream) {
    DOMINO_API_RANGE();
    int rc = ready_for_compute(h);
    if (rc) return rc;
    if (!next_dev && !mask_dev) return DOMINO_E_INVALID_ARG;
    if (h->stack) return DOMINO_E_UNSUPPORTED;
    DeviceGuard g(h->device);
    StepView v = make_view(h);
    if (use_tree(h)) {
        return cuda_status(launch_trie_step(v, make_trie_view(h), h->env, false, h->t_mode, nullptr, nullptr, h->Q,
                                            true, mask_dev, next_dev, (cudaStream_t)stream, nullptr, nullptr,
                                            (int32_t*)h->d_trow.p));
    }
    const int mode = choose_mode(h, v, next_dev != nullptr);
    return cuda_status(launch_step_mask(v, h->env, false, mode, nullptr, nullptr, h->Q, true, mask_dev, next_dev,
                                        (cudaStream_t)stream));
}

int domino_mask_logits(domino_t h, const void* logits_dev, int32_t dtype, int32_t batch,
                       int64_t row_stride_elems, const uint32_t* mask_dev, int32_t* argmax_dev, float* lse_dev,
                       float* logprobs_dev, void* stream) {
    DOMINO_API_RANGE();
    if (!h) return DOMINO_E_INVALID_ARG;
    if (is_host_only(h)) return DOMINO_E_NO_DEVICE;
    if (!h->vocab_loaded) return DOMINO_E_NOT_LOADED;
    if (dtype != DOMINO_DTYPE_F32 && dtype != DOMINO_DTYPE_BF16) return DOMINO_E_INVALID_ARG;
    if (batch < 0 || row_stride_elems < h->V) return DOMINO_E_INVALID_ARG;
    if (batch == 0) return DOMINO_OK;
    if (!logits_dev || !mask_dev || !argmax_dev) return DOMINO_E_INVALID_ARG;
    DeviceGuard g(h->device);
    return cuda_status(launch_mask_logits(h->env, logits_dev, dtype, batch, row_stride_elems, h->V, mask_dev,
                                          argmax_dev, lse_dev, logprobs_dev, (float4*)h->d_partials.p,
                                          (uint32_t*)h->d_counters.p, (float*)h->d_lse_tmp.p,
                                          (cudaStream_t)stream));
}

int domino_advance(domino_t h, const int32_t* states_dev, const uint64_t* stacks_dev, const int32_t* tokens_dev,
                   int32_t batch, int32_t* states_out, uint64_t* stacks_out, void* stream) {
    DOMINO_API_RANGE();
    int rc = ready_for_compute(h);
    if (rc) return rc;
    if (batch < 0) return DOMINO_E_INVALID_ARG;
    if (batch == 0) return DOMINO_OK;
    if (!states_dev || !tokens_dev || !states_out || (stacks_dev && !stacks_out)) return DOMINO_E_INVALID_ARG;
    DeviceGuard g(h->device);
    StepView v = make_view(h);
    const int mode = choose_mode(h, v, false);
    return cuda_status(launch_advance(v, h->stack, mode, states_dev, stacks_dev, tokens_dev, batch, states_out,
                                      stacks_out, (cudaStream_t)stream));
}

int domino_step_decode(domino_t h, const int32_t* states_dev, const uint64_t* stacks_dev, int32_t batch,
                       const void* logits_dev, int32_t dtype, int64_t row_stride_elems, uint32_t* mask_dev,
                       int32_t* argmax_dev, float* lse_dev, float* logprobs_dev, int32_t* states_out,
                       uint64_t* stacks_out, void* stream) {
    DOMINO_API_RANGE();
    int rc = ready_for_compute(h);
    if (rc) return rc;
    if (dtype != DOMINO_DTYPE_F32 && dtype != DOMINO_DTYPE_BF16) return DOMINO_E_INVALID_ARG;
    if (batch < 0 || row_stride_elems < h->V) return DOMINO_E_INVALID_ARG;
    if (batch == 0) return DOMINO_OK;
    if (!states_dev || !logits_dev || !mask_dev || !argmax_dev || (logprobs_dev && !lse_dev) ||
        (states_out && stacks_dev && !stacks_out))
        return DOMINO_E_INVALID_ARG;
    DeviceGuard g(h->device);
    cudaStream_t st = (cudaStream_t)stream;
    // logits in device memory are pulled into L2 a tile ahead of their fold;
    // host-resident logits are read only where the mask allows a token
    cudaPointerAttributes pa{};
    const bool on_device = cudaPointerGetAttributes(&pa, logits_dev) == cudaSuccess && pa.type == cudaMemoryTypeDevice;
    if (!on_device) cudaGetLastError();
    // the fold rides on the per-token walk; where the prefix-tree walk is the
    // faster mask step and the logits sit in device memory, the tree walk, the
    // logits pass and the update run one after the other instead
    const bool fusable = dtype == DOMINO_DTYPE_BF16 && reinterpret_cast<uintptr_t>(logits_dev) % 16 == 0 &&
                         ((size_t)row_stride_elems * 2) % 16 == 0 &&
                         (int64_t)batch * h->n_windows < (int64_t)INT32_MAX &&   // partial slots are int
                         !(on_device && use_tree(h));
    if (!fusable) {   // the kernels one after the other
        if ((rc = domino_step_mask(h, states_dev, stacks_dev, batch, mask_dev, nullptr, stream))) return rc;
        if ((rc = domino_mask_logits(h, logits_dev, dtype, batch, row_stride_elems, mask_dev, argmax_dev, lse_dev,
                                     logprobs_dev, stream)))
            return rc;
        if (!states_out) return DOMINO_OK;
        return domino_advance(h, states_dev, stacks_dev, argmax_dev, batch, states_out, stacks_dev ? stacks_out : nullptr,
                              stream);
    }
    StepView v = make_view(h);
    const size_t part_bytes = (size_t)batch * (size_t)h->n_windows * sizeof(float4);
    if (h->d_fpart.n < part_bytes) {
        // growing the partials buffer synchronises the stream and reallocates,
        // neither of which a stream capture allows: the first call at a larger
        // batch must run uncaptured
        cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
        if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) return cuda_status(cudaGetLastError());
        if (cs != cudaStreamCaptureStatusNone) return DOMINO_E_INVALID_ARG;
        if (cudaStreamSynchronize(st) != cudaSuccess) return cuda_status(cudaGetLastError());
        clear_host_graphs(h);   // recorded host-buffer steps name this buffer
        if ((rc = dev_reserve(h->d_fpart, part_bytes))) return rc;
    }
    const int mode = choose_mode(h, v, false);
    cudaError_t e = launch_step_mask(v, h->env, h->stack, mode, states_dev, stacks_dev, batch, false, mask_dev, nullptr,
                                     st, nullptr, nullptr, logits_dev, row_stride_elems, (float4*)h->d_fpart.p,
                                     on_device);
    if (e == cudaSuccess)
        e = launch_fused_combine(v, h->stack, mode, (const float4*)h->d_fpart.p, batch, h->n_windows, argmax_dev,
                                 lse_dev, states_dev, stacks_dev, states_out, stacks_dev ? stacks_out : nullptr, st);
    if (e == cudaSuccess && logprobs_dev)
        e = launch_logprobs_bf16(h->env, logits_dev, batch, row_stride_elems, h->V, mask_dev, lse_dev, logprobs_dev,
                                 st);
    return cuda_status(e);
}

int domino_mask_sample(domino_t h, const void* logits_dev, int32_t dtype, int32_t batch, int64_t row_stride_elems,
                       const uint32_t* mask_dev, float temperature, uint64_t seed, uint64_t offset,
                       int32_t* tokens_dev, void* stream) {
    DOMINO_API_RANGE();
    if (!h) return DOMINO_E_INVALID_ARG;
    if (is_host_only(h)) return DOMINO_E_NO_DEVICE;
    if (!h->vocab_loaded) return DOMINO_E_NOT_LOADED;
    if (dtype != DOMINO_DTYPE_F32 && dtype != DOMINO_DTYPE_BF16) return DOMINO_E_INVALID_ARG;
    if (!(temperature > 0.0f) || !std::isfinite(temperature) || !std::isfinite(1.0f / temperature))
        return DOMINO_E_INVALID_ARG;
    if (batch < 0 || row_stride_elems < h->V) return DOMINO_E_INVALID_ARG;
    if (batch == 0) return DOMINO_OK;
    if (!logits_dev || !mask_dev || !tokens_dev) return DOMINO_E_INVALID_ARG;
    DeviceGuard g(h->device);
    return cuda_status(launch_mask_sample(h->env, logits_dev, dtype, batch, row_stride_elems, h->V, mask_dev,
                                          temperature, seed, offset, tokens_dev, (float4*)h->d_partials.p,
                                          (uint32_t*)h->d_counters.p, (cudaStream_t)stream));
}

int domino_opportunistic_step(domino_t h, const void* logits_dev, int32_t dtype, int32_t batch,
                              int64_t row_stride_elems, const int32_t* states_dev, const uint64_t* stacks_dev,
                              uint32_t* mask_scratch_dev, int32_t* tokens_dev, int32_t* n_fallback_dev,
                              void* stream) {
    DOMINO_API_RANGE();
    int rc = ready_for_compute(h);
    if (rc) return rc;
    if (dtype != DOMINO_DTYPE_F32 && dtype != DOMINO_DTYPE_BF16) return DOMINO_E_INVALID_ARG;
    if (batch < 0 || row_stride_elems < h->V) return DOMINO_E_INVALID_ARG;
    if (batch == 0) return DOMINO_OK;
    if (!logits_dev || !states_dev || !mask_scratch_dev || !tokens_dev) return DOMINO_E_INVALID_ARG;
    DeviceGuard g(h->device);
    cudaStream_t st = (cudaStream_t)stream;
    if (h->o_prop.n < (size_t)batch * 4 || h->o_rows.n < (size_t)batch * 4 || h->o_count.n < 16) {
        if (cudaStreamSynchronize(st) != cudaSuccess) return cuda_status(cudaGetLastError());
        if ((rc = dev_reserve(h->o_prop, (size_t)batch * 4))) return rc;
        if ((rc = dev_reserve(h->o_rows, (size_t)batch * 4))) return rc;
        if ((rc = dev_reserve(h->o_count, 16))) return rc;
    }
    int32_t* prop = (int32_t*)h->o_prop.p;
    int32_t* rows = (int32_t*)h->o_rows.p;
    int32_t* count = n_fallback_dev ? n_fallback_dev : (int32_t*)h->o_count.p;
    StepView v = make_view(h);
    const int mode = choose_mode(h, v, false);
    cudaError_t e = cudaMemsetAsync(count, 0, sizeof(int32_t), st);
    // 1. the unmasked argmax (every token allowed)
    if (e == cudaSuccess)
        e = launch_mask_logits(h->env, logits_dev, dtype, batch, row_stride_elems, h->V, nullptr, prop, nullptr,
                               nullptr, (float4*)h->d_partials.p, (uint32_t*)h->d_counters.p, nullptr, st);
    // 2. one walk per row: keep the proposal or list the row for the fallback
    if (e == cudaSuccess)
        e = launch_propose_check(v, h->stack, mode, states_dev, stacks_dev, prop, batch, tokens_dev, rows, count, st);
    // 3. the listed rows only: their masks, then their masked argmax
    if (e == cudaSuccess)
        e = launch_step_mask(v, h->env, h->stack, mode, states_dev, stacks_dev, batch, false, mask_scratch_dev,
                             nullptr, st, rows, count);
    if (e == cudaSuccess)
        e = launch_mask_logits(h->env, logits_dev, dtype, batch, row_stride_elems, h->V, mask_scratch_dev,
                               tokens_dev, nullptr, nullptr, (float4*)h->d_partials.p, (uint32_t*)h->d_counters.p,
                               nullptr, st, nullptr, 0, nullptr, nullptr, rows, count);
    return cuda_status(e);
}

int domino_spec_update(domino_t h, uint32_t* counts_dev, uint64_t* best_dev, uint32_t* reached_dev,
                       const int32_t* states_dev, const uint64_t* stacks_dev, const int32_t* tokens_dev,
                       int32_t batch, void* stream) {
    DOMINO_API_RANGE();
    int rc = ready_for_compute(h);
    if (rc) return rc;
    if (batch < 0) return DOMINO_E_INVALID_ARG;
    if (batch == 0) return DOMINO_OK;
    if (!counts_dev || !best_dev || !reached_dev || !states_dev || !tokens_dev) return DOMINO_E_INVALID_ARG;
    DeviceGuard g(h->device);
    StepView v = make_view(h);
    return cuda_status(launch_spec_update(v, h->stack, states_dev, stacks_dev, tokens_dev, batch, counts_dev,
                                          (unsigned long long*)best_dev, reached_dev, (cudaStream_t)stream));
}

int domino_spec_propose(domino_t h, const uint64_t* best_dev, const uint32_t* reached_dev,
                        const int32_t* states_dev, const uint64_t* stacks_dev, int32_t batch, int32_t s,
                        int32_t min_permille, int32_t* proposals_dev, int32_t* n_prop_dev,
                        int32_t* chain_states_dev, uint64_t* chain_stacks_dev, void* stream) {
    DOMINO_API_RANGE();
    int rc = ready_for_compute(h);
    if (rc) return rc;
    if (batch < 0 || s < 1 || min_permille < 0 || min_permille > 1000) return DOMINO_E_INVALID_ARG;
    if (batch == 0) return DOMINO_OK;
    if (!best_dev || !reached_dev || !states_dev || !proposals_dev || !n_prop_dev || !chain_states_dev)
        return DOMINO_E_INVALID_ARG;
    if (stacks_dev && !chain_stacks_dev) return DOMINO_E_INVALID_ARG;
    DeviceGuard g(h->device);
    StepView v = make_view(h);
    const int mode = choose_mode(h, v, false);
    return cuda_status(launch_spec_propose(v, h->stack, mode, states_dev, stacks_dev, batch, s, min_permille,
                                           (const unsigned long long*)best_dev, reached_dev, proposals_dev,
                                           n_prop_dev, chain_states_dev, chain_stacks_dev, (cudaStream_t)stream));
}

int domino_spec_accept(domino_t h, const int32_t* proposals_dev, const int32_t* n_prop_dev,
                       const int32_t* decoded_dev, const int32_t* chain_states_dev, const uint64_t* chain_stacks_dev,
                       int32_t batch, int32_t s, int32_t* n_accept_dev, int32_t* tokens_out_dev,
                       int32_t* states_out_dev, uint64_t* stacks_out_dev, void* stream) {
    DOMINO_API_RANGE();
    if (!h) return DOMINO_E_INVALID_ARG;
    if (is_host_only(h)) return DOMINO_E_NO_DEVICE;
    if (batch < 0 || s < 1) return DOMINO_E_INVALID_ARG;
    if (batch == 0) return DOMINO_OK;
    if (!proposals_dev || !n_prop_dev || !decoded_dev || !n_accept_dev) return DOMINO_E_INVALID_ARG;
    if ((states_out_dev && !chain_states_dev) || (stacks_out_dev && !chain_stacks_dev)) return DOMINO_E_INVALID_ARG;
    DeviceGuard g(h->device);
    return cuda_status(launch_spec_accept(proposals_dev, n_prop_dev, decoded_dev, chain_states_dev, chain_stacks_dev,
                                          batch, s, n_accept_dev, tokens_out_dev, states_out_dev, stacks_out_dev,
                                          (cudaStream_t)stream));
}

int domino_mask_logits_table(domino_t h, const void* logits_dev, int32_t dtype, int32_t batch,
                             int64_t row_stride_elems, const uint32_t* table_mask_dev, const int32_t* states_dev,
                             int32_t* argmax_dev, float* lse_dev, float* logprobs_dev, void* stream) {
    DOMINO_API_RANGE();
    int rc = ready_for_compute(h);
    if (rc) return rc;
    if (h->stack) return DOMINO_E_UNSUPPORTED;
    if (dtype != DOMINO_DTYPE_F32 && dtype != DOMINO_DTYPE_BF16) return DOMINO_E_INVALID_ARG;
    if (batch < 0 || row_stride_elems < h->V) return DOMINO_E_INVALID_ARG;
    if (batch == 0) return DOMINO_OK;
    if (!logits_dev || !table_mask_dev || !states_dev || !argmax_dev) return DOMINO_E_INVALID_ARG;
    DeviceGuard g(h->device);
    return cuda_status(launch_mask_logits(h->env, logits_dev, dtype, batch, row_stride_elems, h->V, table_mask_dev,
                                          argmax_dev, lse_dev, logprobs_dev, (float4*)h->d_partials.p,
                                          (uint32_t*)h->d_counters.p, (float*)h->d_lse_tmp.p, (cudaStream_t)stream,
                                          states_dev, h->Q, (uint32_t*)h->d_err.p));
}

int domino_advance_table(domino_t h, const int32_t* table_next_dev, const int32_t* states_dev,
                         const int32_t* tokens_dev, int32_t batch, int32_t* states_out, void* stream) {
    DOMINO_API_RANGE();
    int rc = ready_for_compute(h);
    if (rc) return rc;
    if (h->stack) return DOMINO_E_UNSUPPORTED;
    if (batch < 0) return DOMINO_E_INVALID_ARG;
    if (batch == 0) return DOMINO_OK;
    if (!table_next_dev || !states_dev || !tokens_dev || !states_out) return DOMINO_E_INVALID_ARG;
    DeviceGuard g(h->device);
    return cuda_status(launch_advance_table(table_next_dev, h->Q, h->V, h->eos_id, h->start, states_dev, tokens_dev,
                                            batch, states_out, (uint32_t*)h->d_err.p, (cudaStream_t)stream));
}

namespace {

// The host-buffer step's small inputs and outputs in one buffer (device s_io,
// pinned host h_io): [tokens | lse | states | stacks], each part on a 16-byte
// boundary.  The copy path moves states and stacks up in one copy and
// everything back in one; the in-place path's kernels read and write h_io
// directly.
struct IoLayout {
    size_t tok, lse, st, sk, in_end;
};
IoLayout io_layout(int32_t batch, bool stacks) {
    auto a16 = [](size_t x) { return (x + 15) / 16 * 16; };
    IoLayout L{};
    L.tok = 0;
    L.lse = a16(L.tok + (size_t)batch * 4);
    L.st = a16(L.lse + (size_t)batch * 4);
    L.sk = a16(L.st + (size_t)batch * 4);
    L.in_end = stacks ? L.sk + (size_t)batch * 8 : L.st + (size_t)batch * 4;
    return L;
}

// Pageable logits: the configurations and then the logits are copied in up
// to 8 chunks of rows on the copy stream; the mask step runs while they copy,
// and each chunk's masked argmax starts as soon as its rows have landed.
int copy_and_decode_chunks(domino_ctx* h, const void* logits_host, int32_t dtype, int32_t batch, bool stacks,
                           const IoLayout& L, cudaStream_t st) {
    int rc;
    void* stream = (void*)st;
    const size_t esz = dtype == DOMINO_DTYPE_BF16 ? 2 : 4;
    const size_t row_bytes = (size_t)h->V * esz;
    const size_t logit_bytes = (size_t)batch * row_bytes;
    char* io = (char*)h->s_io.p;
    int32_t* d_states = (int32_t*)(io + L.st);
    uint64_t* d_stacks = stacks ? (uint64_t*)(io + L.sk) : nullptr;
    uint32_t* d_mask = (uint32_t*)h->s_mask.p;
    int32_t* d_tok = (int32_t*)(io + L.tok);
    float* d_lse = (float*)(io + L.lse);
    const int n_chunks = (int)std::max<size_t>(1, std::min<size_t>({(size_t)8, (size_t)batch, logit_bytes >> 23}));
    cudaError_t e = cudaEventRecord(h->ev_cfg, st);   // the caller's earlier work on `stream` comes first
    if (e == cudaSuccess) e = cudaStreamWaitEvent(h->cp_stream, h->ev_cfg, 0);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(io + L.st, (char*)h->h_io + L.st, L.in_end - L.st, cudaMemcpyHostToDevice, h->cp_stream);
    if (e == cudaSuccess) e = cudaEventRecord(h->ev_cfg, h->cp_stream);
    std::vector<int32_t> r0s((size_t)n_chunks + 1);
    for (int k = 0; k <= n_chunks; ++k) r0s[(size_t)k] = (int32_t)(((int64_t)batch * k) / n_chunks);
    if (e == cudaSuccess) e = cudaEventRecord(h->ev_t[2], h->cp_stream);
    for (int k = 0; k < n_chunks && e == cudaSuccess; ++k) {
        const size_t off = (size_t)r0s[(size_t)k] * row_bytes, n = (size_t)(r0s[(size_t)k + 1] - r0s[(size_t)k]) * row_bytes;
        e = cudaMemcpyAsync((char*)h->s_logits.p + off, (const char*)logits_host + off, n, cudaMemcpyHostToDevice,
                            h->cp_stream);
        if (e == cudaSuccess) e = cudaEventRecord(h->ev_chunk[k], h->cp_stream);
    }
    if (e == cudaSuccess) e = cudaEventRecord(h->ev_t[3], h->cp_stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(st, h->ev_cfg, 0);
    if (e != cudaSuccess) return cuda_status(e);
    if ((rc = domino_step_mask(h, d_states, d_stacks, batch, d_mask, nullptr, stream))) return rc;
    for (int k = 0; k < n_chunks; ++k) {
        const int32_t r0 = r0s[(size_t)k], rows = r0s[(size_t)k + 1] - r0;
        if ((e = cudaStreamWaitEvent(st, h->ev_chunk[k], 0)) != cudaSuccess) return cuda_status(e);
        if ((rc = domino_mask_logits(h, (const char*)h->s_logits.p + (size_t)r0 * row_bytes, dtype, rows, h->V,
                                     d_mask + (size_t)r0 * h->W, d_tok + r0, d_lse + r0, nullptr, stream)))
            return rc;
    }
    // every copy-stream node rejoins `stream` (a recorded graph needs it; the
    // copies are done by now anyway)
    return cuda_status(cudaStreamWaitEvent(st, h->ev_t[3], 0));
}

// The host-buffer step's copies and launches on `st` (and the copy stream),
// without the final synchronisation.  The states and stacks are already in
// h_io; the outputs land there.
int enqueue_host_step(domino_ctx* h, const void* logits_host, void* logits_mapped, bool mapped, int32_t dtype,
                      int32_t batch, bool stacks, const IoLayout& L, cudaStream_t st) {
    int rc;
    void* stream = (void*)st;
    char* io = (char*)h->s_io.p;
    int32_t* d_states = (int32_t*)(io + L.st);
    uint64_t* d_stacks = stacks ? (uint64_t*)(io + L.sk) : nullptr;
    uint32_t* d_mask = (uint32_t*)h->s_mask.p;
    int32_t* d_tok = (int32_t*)(io + L.tok);
    float* d_lse = (float*)(io + L.lse);
    if (mapped) {
        // the mask step folds the pinned logits it allows, read in place; the
        // configurations are read from and the results written to the pinned
        // staging buffer itself (no copies: two kernels)
        char* hio = (char*)h->h_io_dev;
        int32_t* m_states = (int32_t*)(hio + L.st);
        uint64_t* m_stacks = stacks ? (uint64_t*)(hio + L.sk) : nullptr;
        return domino_step_decode(h, m_states, m_stacks, batch, logits_mapped, dtype, h->V, d_mask,
                                  (int32_t*)(hio + L.tok), (float*)(hio + L.lse), nullptr, m_states, m_stacks, stream);
    } else {
        if ((rc = copy_and_decode_chunks(h, logits_host, dtype, batch, stacks, L, st))) return rc;
        if ((rc = domino_advance(h, d_states, d_stacks, d_tok, batch, d_states, d_stacks, stream))) return rc;
    }
    return cuda_status(cudaMemcpyAsync(h->h_io, io, L.in_end, cudaMemcpyDeviceToHost, st));
}

}  // namespace

int domino_decode_step_host(domino_t h, const void* logits_host, int32_t dtype, int32_t batch,
                            int32_t* states_host, uint64_t* stacks_host, int32_t* tokens_host, float* lse_host,
                            void* stream) {
    DOMINO_API_RANGE();
    int rc = ready_for_compute(h);
    if (rc) return rc;
    if (dtype != DOMINO_DTYPE_F32 && dtype != DOMINO_DTYPE_BF16) return DOMINO_E_INVALID_ARG;
    if (batch < 0) return DOMINO_E_INVALID_ARG;
    if (batch == 0) return DOMINO_OK;
    if (!logits_host || !states_host || !tokens_host) return DOMINO_E_INVALID_ARG;
    DeviceGuard g(h->device);
    cudaStream_t st = (cudaStream_t)stream;
    const size_t esz = dtype == DOMINO_DTYPE_BF16 ? 2 : 4;
    const size_t row_bytes = (size_t)h->V * esz;
    const size_t logit_bytes = (size_t)batch * row_bytes;
    const bool stacks = stacks_host != nullptr;
    const IoLayout L = io_layout(batch, stacks);
    // Pinned (page-locked, mapped) bf16 logits can be read where they are: the
    // mask step folds each tile's allowed logits, so only those cross the host
    // link, while the walk runs.  Or they are copied in chunks while the mask
    // step runs and decoded as they land.  Which is faster depends on the
    // masks' density and on the link's read granularity, so it is measured:
    // each path's host wall time is averaged over settled calls (no buffer growth,
    // no recording), the faster one is used, and every 64th call takes the
    // other to keep its time current.
    const auto t_enter = std::chrono::steady_clock::now();
    cudaPointerAttributes pa{};
    const bool pinned = cudaPointerGetAttributes(&pa, logits_host) == cudaSuccess && pa.type == cudaMemoryTypeHost &&
                        pa.devicePointer != nullptr;
    if (!pinned) cudaGetLastError();
    bool mapped = pinned && dtype == DOMINO_DTYPE_BF16;
    const bool choice = mapped;
    if (choice) {
        if (h->t_wall_ms[1] == 0.0) mapped = true;
        else if (h->t_wall_ms[0] == 0.0) mapped = false;
        else mapped = (h->t_wall_ms[1] <= h->t_wall_ms[0]) != (h->host_calls % 64 == 63);
    }
    // the in-place path runs the fused decode, whose per-window partials
    // buffer is grown here too, before any recording
    const size_t fpart_bytes = (size_t)batch * (size_t)h->n_windows * sizeof(float4);
    const bool grow = (!mapped && h->s_logits.n < logit_bytes) || h->s_io.n < L.in_end ||
                      h->s_mask.n < (size_t)batch * (size_t)h->W * 4 || h->h_io_n < L.in_end || !h->cp_stream ||
                      (mapped && h->d_fpart.n < fpart_bytes);
    if (grow) {   // buffers may move: recorded steps that use them are dropped
        if (cudaStreamSynchronize(st) != cudaSuccess) return cuda_status(cudaGetLastError());
        clear_host_graphs(h);
    }
    if (!mapped && (rc = dev_reserve(h->s_logits, logit_bytes))) return rc;
    if (mapped && (rc = dev_reserve(h->d_fpart, fpart_bytes))) return rc;
    if ((rc = dev_reserve(h->s_mask, (size_t)batch * (size_t)h->W * 4))) return rc;
    if ((rc = dev_reserve(h->s_io, L.in_end))) return rc;
    if (h->h_io_n < L.in_end) {
        if (h->h_io) cudaFreeHost(h->h_io);
        h->h_io = nullptr;
        h->h_io_n = 0;
        if (cudaMallocHost(&h->h_io, L.in_end) != cudaSuccess) {
            cudaGetLastError();
            h->h_io = nullptr;
            return DOMINO_E_OOM;
        }
        if (cudaHostGetDevicePointer(&h->h_io_dev, h->h_io, 0) != cudaSuccess) {
            cudaGetLastError();
            cudaFreeHost(h->h_io);
            h->h_io = h->h_io_dev = nullptr;
            return DOMINO_E_CUDA;
        }
        h->h_io_n = L.in_end;
    }
    if (!h->cp_stream) {
        cudaError_t e = cudaStreamCreateWithFlags(&h->cp_stream, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_cfg, cudaEventDisableTiming);
        for (cudaEvent_t& ev : h->ev_chunk)
            if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
        for (cudaEvent_t& ev : h->ev_t)
            if (e == cudaSuccess) e = cudaEventCreate(&ev);
        if (e != cudaSuccess) return cuda_status(e);
    }
    std::memcpy((char*)h->h_io + L.st, states_host, (size_t)batch * 4);
    if (stacks) std::memcpy((char*)h->h_io + L.sk, stacks_host, (size_t)batch * 8);
    // The step's copies and launches, recorded once per set of buffers and
    // path on a non-default stream (the default stream cannot be captured) and
    // replayed afterwards.  The first two calls of a handle run them directly
    // (the first sets kernel attributes).
    const void* key[16] = {logits_host, (const void*)(intptr_t)batch,
                           (const void*)(intptr_t)(dtype * 4 + (mapped ? 1 : 0) + (stacks ? 2 : 0)), h->s_logits.p,
                           h->s_mask.p, h->s_io.p, h->h_io, (const void*)st, nullptr, nullptr, nullptr, nullptr,
                           nullptr, nullptr, nullptr, nullptr};
    cudaGraphExec_t exec = nullptr;
    for (auto& hg : h->host_graphs)
        if (std::equal(std::begin(key), std::end(key), std::begin(hg.key))) {
            exec = hg.exec;
            hg.used = h->host_calls;
        }
    cudaError_t e = cudaSuccess;
    const bool record = !exec && st != nullptr && h->host_calls > 1;
    if (record) {
        cudaGraph_t gr = nullptr;
        e = cudaStreamBeginCapture(st, cudaStreamCaptureModeRelaxed);
        if (e != cudaSuccess) return cuda_status(e);
        rc = enqueue_host_step(h, logits_host, pa.devicePointer, mapped, dtype, batch, stacks, L, st);
        e = cudaStreamEndCapture(st, &gr);
        if (rc || e != cudaSuccess) {
            if (gr) cudaGraphDestroy(gr);
            return rc ? rc : cuda_status(e);
        }
        e = cudaGraphInstantiate(&exec, gr, 0);
        cudaGraphDestroy(gr);
        if (e != cudaSuccess) return cuda_status(e);
        if (h->host_graphs.size() >= 8) {   // keep the 8 most recently used
            auto lru = std::min_element(h->host_graphs.begin(), h->host_graphs.end(),
                                        [](const domino_ctx::HostGraph& x, const domino_ctx::HostGraph& y) {
                                            return x.used < y.used;
                                        });
            cudaGraphExecDestroy(lru->exec);
            h->host_graphs.erase(lru);
        }
        domino_ctx::HostGraph hg{};
        std::copy(std::begin(key), std::end(key), std::begin(hg.key));
        hg.exec = exec;
        hg.used = h->host_calls;
        h->host_graphs.push_back(hg);
    }
    if (exec) {
        e = cudaGraphLaunch(exec, st);
    } else if ((rc = enqueue_host_step(h, logits_host, pa.devicePointer, mapped, dtype, batch, stacks, L, st))) {
        return rc;
    }
    h->host_calls++;
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_status(e);
    const char* io = (const char*)h->h_io;
    std::memcpy(tokens_host, io + L.tok, (size_t)batch * 4);
    if (lse_host) std::memcpy(lse_host, io + L.lse, (size_t)batch * 4);
    std::memcpy(states_host, io + L.st, (size_t)batch * 4);
    if (stacks) std::memcpy(stacks_host, io + L.sk, (size_t)batch * 8);
    if (choice && !grow && !record && h->host_calls > 1) {
        // a moving average, so that one slow call (the host preempted, a
        // shared link) does not send the next 64 calls down the slower path
        const double t = std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t_enter).count();
        double& avg = h->t_wall_ms[mapped ? 1 : 0];
        avg = avg == 0.0 ? t : 0.75 * avg + 0.25 * t;
    }
    return DOMINO_OK;
}


int domino_get_device_error(domino_t h, int32_t* code, void* stream) {
    if (!h || !code) return DOMINO_E_INVALID_ARG;
    *code = 0;
    if (is_host_only(h)) return DOMINO_E_NO_DEVICE;
    DeviceGuard g(h->device);
    cudaStream_t st = (cudaStream_t)stream;
    uint32_t word = 0;
    cudaError_t e = cudaMemcpyAsync(&word, h->d_err.p, 4, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaMemsetAsync(h->d_err.p, 0, 4, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_status(e);
    *code = (int32_t)word;
    return DOMINO_OK;
}

}  // extern "C"
