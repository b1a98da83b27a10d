"""The prefix tree the mask step walks (Alg. 2's subterminal tree over byte
classes, Sec. 3.3), checked on the CPU through a host-only handle:

- structure: preorder numbering, nested token ranges, every token of the
  vocabulary except EOS and empty tokens exactly once, at the node whose path
  spells its class string; children in class order; the classes-below sets;
  the upper nodes (large subtrees) and the units (the subtrees hanging off
  them) cover every node once;
- a model of the two kernels over the exported arrays (each row's
  configuration at the upper nodes, then one walk per live (row, unit) pair
  with a stack of at most kTrieBranch entries) gives the oracle's masks and
  next states on workload rows.
"""
import numpy as np
import pytest

from paper_2403_06988_gb300 import synth

B = pytest.importorskip("paper_2403_06988_gb300._binding")

TRIE_BRANCH = 8          # kTrieBranch: the walk's stack bound
TRIE_TILE = 64           # kTrieTile: the largest unit


def host_handle(a, v):
    h = B.domino_create(-1)
    B.domino_load_vocab(h, v.data, v.offsets, v.n_tokens, v.eos_id)
    B.domino_load_automaton(h, a.delta, a.n_states, a.live, a.accepting, a.start, a.rules, None, a.max_depth)
    return h


def tree_of(a, v):
    h = host_handle(a, v)
    try:
        nodes, toks, upper, units = B.domino_get_prefix_tree(h)
        cls = B.domino_get_byte_classes(h)
        K = int(cls.max()) + 1
    finally:
        B.domino_destroy(h)
    return nodes, toks, upper, units, cls, K


def children(nodes, n):
    c = n + 1
    end = int(nodes[n, 0] & 0xFFFFFF)
    while c < end:
        yield c
        c = int(nodes[c, 0] & 0xFFFFFF)


def check_structure(a, v):
    nodes, toks, upper, units, cls, K = tree_of(a, v)
    N = nodes.shape[0]
    skip = (nodes[:, 0] & 0xFFFFFF).astype(np.int64)
    ncls = (nodes[:, 0] >> 24).astype(np.int64)
    tok_lo, n_end, tok_hi = nodes[:, 1].astype(np.int64), nodes[:, 2].astype(np.int64), nodes[:, 3].astype(np.int64)
    assert skip[0] == N and tok_lo[0] == 0 and n_end[0] == 0 and tok_hi[0] == len(toks)
    assert (skip > np.arange(N)).all() and (skip <= N).all()
    # every token but EOS and empty ones, once
    tl = v.tokens()
    want = sorted(t for t in range(v.n_tokens) if t != v.eos_id and len(tl[t]) > 0)
    assert sorted(toks.tolist()) == want
    # paths, ranges, child order, classes below, branching heights
    path = {0: b""}
    sub = np.zeros(N, dtype=object)
    bh = np.zeros(N, np.int64)
    parent = np.zeros(N, np.int64)
    for n in range(N - 1, -1, -1):
        m, hmax, k = 0, 0, 0
        for c in children(nodes, n):
            m |= (1 << int(ncls[c])) | int(sub[c])
            hmax = max(hmax, bh[c])
            k += 1
            parent[c] = n
        sub[n] = m
        bh[n] = hmax + (1 if k >= 2 else 0)
    for n in range(N):
        assert tok_lo[n] + n_end[n] <= tok_hi[n]
        cs = list(children(nodes, n))
        assert [int(ncls[c]) for c in cs] == sorted(set(int(ncls[c]) for c in cs))   # strictly increasing
        expect_lo = tok_lo[n] + n_end[n]
        for c in cs:
            path[c] = path[n] + bytes([int(ncls[c])])
            assert tok_lo[c] == expect_lo
            expect_lo = tok_hi[c]
        assert expect_lo == tok_hi[n]
        for t in toks[tok_lo[n]:tok_lo[n] + n_end[n]]:
            assert bytes(cls[np.frombuffer(tl[t], np.uint8)]) == path[n]
        if K <= 64:
            got = int(nodes[n, 4]) | (int(nodes[n, 5]) << 32)
            assert got == sub[n]
    # upper nodes: the root and the nodes with large subtrees, in preorder
    is_up = np.zeros(N, bool)
    is_up[0] = True
    is_up |= (skip - np.arange(N) > TRIE_TILE) | (bh > TRIE_BRANCH)
    assert upper[:, 0].tolist() == np.flatnonzero(is_up).tolist()
    for u, d in upper.tolist():
        assert d == len(path[u])
    # units: every non-upper node whose parent is upper, with that parent's index
    uidx = {int(n): i for i, n in enumerate(upper[:, 0].tolist())}
    roots = [n for n in range(1, N) if not is_up[n] and is_up[parent[n]]]
    assert units[:, 0].tolist() == roots
    assert units[:, 1].tolist() == [uidx[int(parent[n])] for n in roots]
    covered = np.zeros(N, np.int64)
    covered[is_up] += 1
    for r in roots:
        covered[r:skip[r]] += 1
    assert (covered == 1).all()
    return nodes, toks, upper, units, cls, K


@pytest.mark.parametrize("config", [1, 2, 5])
def test_tree_structure_workloads(config):
    w = synth.workload(config)
    check_structure(w.automaton, w.vocab)


def test_tree_structure_ragged_vocab_with_duplicate_class_strings():
    a = synth.int_regex_dfa()
    rng = np.random.default_rng(8)
    toks = set()
    while len(toks) < 1500:
        toks.add(rng.choice(np.frombuffer(b"-0123456789x", np.uint8), int(rng.integers(1, 40))).tobytes())
    toks = sorted(toks)
    toks.insert(300, b"")          # EOS
    toks.insert(900, b"")          # an empty token that is not EOS
    v = synth.Vocab.from_tokens(toks, eos_id=300)
    nodes, *_ = check_structure(a, v)
    assert nodes.shape[0] > 100


# --------------------------------------------------------------------------
# a model of the kernel's traversal
# --------------------------------------------------------------------------
class Model:
    def __init__(self, a, v):
        (self.nodes, self.toks, self.upper, self.units, self.cls, self.K) = tree_of(a, v)
        self.a, self.v = a, v
        self.rep = np.zeros(self.K, np.int64)
        for b in range(255, -1, -1):
            self.rep[self.cls[b]] = b
        self.rules = {}
        if a.rules is not None:
            for r in a.rules:
                self.rules[(int(r["state"]), int(r["byte"]))] = r
        N = self.nodes.shape[0]
        par = np.zeros(N, np.int64)
        for n in range(N):
            for c in children(self.nodes, n):
                par[c] = n
        self.upaths = []
        for u, d in self.upper.tolist():
            p, x = [], u
            while x != 0:
                p.append(int(self.nodes[x, 0] >> 24))
                x = int(par[x])
            assert len(p) == d
            self.upaths.append(p[::-1])

    def step(self, cfg, c):
        s, bits, depth = cfg
        b = int(self.rep[c])
        r = self.rules.get((s, b))
        if r is None:
            s2 = int(self.a.delta[s, b])
        elif r["kind"] == synth.RULE_PUSH:
            if depth >= self.a.max_depth:
                return None
            bits, depth, s2 = (bits << 1) | int(r["sym"]), depth + 1, int(self.a.delta[s, b])
        else:
            if depth == 0 or (bits & 1) != int(r["sym"]):
                return None
            bits, depth = bits >> 1, depth - 1
            rev = 0 if depth == 0 else 1 + (bits & 1)
            s2 = int((r["next_if_empty"], r["next_if_top0"], r["next_if_top1"])[rev])
        return (s2, bits, depth) if s2 != 0 and self.a.live[s2] else None

    def row(self, s0, stack_word):
        """mask bits and next states of one row, as the two kernels compute them"""
        V = self.v.n_tokens
        nodes, toks = self.nodes, self.toks
        allowed = {}
        cfg0 = (int(s0), int(stack_word) & 0xFFFFFFFF, int(stack_word) >> 32)
        if self.v.eos_id >= 0 and cfg0[2] == 0 and self.a.accepting[cfg0[0]]:
            allowed[self.v.eos_id] = cfg0[0]
        # the upper kernel: the row's configuration at every upper node
        ucfg = []
        for (u, _), p in zip(self.upper.tolist(), self.upaths):
            cfg = cfg0
            for c in p:
                cfg = self.step(cfg, c) if cfg is not None else None
            ucfg.append(cfg)
            if cfg is not None:
                lo, ne = int(nodes[u, 1]), int(nodes[u, 2])
                for t in toks[lo:lo + ne].tolist():
                    allowed[t] = cfg[0]
        # the tile kernel: one walk per live (unit, row) pair
        for root, pu in self.units.tolist():
            if ucfg[pu] is not None:
                self.walk(root, ucfg[pu], allowed)
        mask = np.zeros((V + 31) // 32, np.uint32)
        nxt_states = np.zeros(V, np.int32)
        for t, s in allowed.items():
            mask[t >> 5] |= np.uint32(1 << (t & 31))
            nxt_states[t] = s
        return mask, nxt_states

    def walk(self, x, cfg, allowed):
        nodes, toks = self.nodes, self.toks
        end = x + 1
        stack = []
        while True:
            while x < end:
                xs = int(nodes[x, 0] & 0xFFFFFF)
                c2 = self.step(cfg, int(nodes[x, 0] >> 24))
                if c2 is not None:
                    lo, ne = int(nodes[x, 1]), int(nodes[x, 2])
                    for t in toks[lo:lo + ne].tolist():
                        allowed[t] = c2[0]
                    if xs > x + 1:
                        if xs < end:
                            stack.append((xs, end, cfg))
                            assert len(stack) <= TRIE_BRANCH
                        x, end, cfg = x + 1, xs, c2
                        continue
                x = xs
            if not stack:
                return
            x, end, cfg = stack.pop()


@pytest.mark.parametrize("config,rows", [(1, None), (2, None), (3, 24), (5, 6)])
def test_traversal_model_matches_oracle(config, rows):
    import oracle
    w = synth.workload(config)
    states, stacks = w.initial_configs()
    if rows is not None:
        states, stacks = states[:rows], stacks[:rows]
    m = Model(w.automaton, w.vocab)
    P = oracle.Problem.from_workload(w)
    has_stack = w.automaton.rules is not None
    m_o, n_o, bad = P.step_mask(states, stacks if has_stack else None, want_next=True)
    assert bad == 0
    for i in range(len(states)):
        mk, nx = m.row(states[i], stacks[i] if has_stack else 0)
        assert (mk == m_o[i]).all(), i
        assert (nx == n_o[i]).all(), i
