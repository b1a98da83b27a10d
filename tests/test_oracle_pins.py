"""Pins for the CPU oracle: what the paper and the mathematics fix, checked
without reusing the oracle's own formulas.

  * Fig. 3 worked example (golden fixture, cited there).
  * Brute force: on tiny grammars, every string up to length N is run through an
    independent recognizer (Python `re`, a recursive-descent parser, a stack
    checker); a token is allowed after prefix u iff u.t is a prefix of some
    member (Definition "minimally invasive", Sec. 2; k = infinity, Sec. 3.5).
  * Invariants: allowed => live next state; rejected => next 0; next-state
    composition over concatenated tokens; stack-depth bounds (Sec. 3.4).
  * Logits: closed forms (uniform, single allowed, ties, all masked) and an
    independent log-sum-exp (scipy) for Alg. 1's masked decode.
"""
import itertools
import math
import os
import re

import numpy as np
import pytest

from paper_2403_06988_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def byte_vocab():
    return synth.Vocab.from_tokens([bytes([c]) for c in range(256)])


def walk_prefix(oracle, automaton, u: bytes):
    """Configuration after the byte string u (None when u is rejected)."""
    P = oracle.Problem.from_parts(automaton, byte_vocab())
    s, w = automaton.start, 0
    for c in u:
        r, s2, w2 = P.check(s, w, c)
        if r != 1:
            return None
        s, w = s2, w2
    return s, w


# --------------------------------------------------------------------------
# Fig. 3 worked example
# --------------------------------------------------------------------------
def read_fig3():
    prefix, cases = None, []
    with open(os.path.join(GOLDEN, "fig3_masks.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            parts = line.rstrip("\n").split("\t")
            if parts[0] == "prefix":
                prefix = parts[1].encode()
            else:
                tok = b"" if parts[1] == "<eos>" else parts[1].replace("\\x20", " ").encode()
                cases.append((tok, parts[2] == "allowed"))
    return prefix, cases


def test_fig3_worked_example(oracle_lib):
    prefix, cases = read_fig3()
    a = synth.fig3_expr_pda()
    v = synth.fig3_vocab()
    toks = v.tokens()
    s, w = walk_prefix(oracle_lib, a, prefix)
    P = oracle_lib.Problem.from_parts(a, v)
    mask, nxt, bad = P.step_mask(np.array([s], np.int32), np.array([w], np.uint64), want_next=True)
    assert bad == 0
    bits = oracle_lib.bits_of(mask[0], v.n_tokens)
    assert len(cases) == len(toks)
    for tok, allowed in cases:
        t = toks.index(tok)
        assert bits[t] == allowed, (tok, allowed)
        assert (nxt[0, t] != 0) == allowed


# --------------------------------------------------------------------------
# brute force against independent recognizers
# --------------------------------------------------------------------------
def expr_member(s: bytes, max_depth: int = 10 ** 9) -> bool:
    """Fig. 3 (a) by recursive descent over a maximal-munch lexer."""
    toks, i, n = [], 0, len(s)
    while i < n:
        c = s[i]
        if c == 0x20:
            i += 1
        elif c in b"()+":
            toks.append(c)
            i += 1
        elif c == 0x30:
            while i < n and s[i] == 0x30:
                i += 1
            toks.append("int")
        elif 0x31 <= c <= 0x39:
            i += 1
            while i < n and 0x30 <= s[i] <= 0x39:
                i += 1
            toks.append("int")
        else:
            return False
    pos = 0

    def term(depth):
        nonlocal pos
        if pos < len(toks) and toks[pos] == "int":
            pos += 1
            return True
        if pos < len(toks) and toks[pos] == ord("("):
            if depth + 1 > max_depth:
                return False
            pos += 1
            if not expr(depth + 1):
                return False
            if pos < len(toks) and toks[pos] == ord(")"):
                pos += 1
                return True
        return False

    def expr(depth):
        nonlocal pos
        if not term(depth):
            return False
        while pos < len(toks) and toks[pos] == ord("+"):
            pos += 1
            if not term(depth):
                return False
        return True

    return expr(0) and pos == len(toks)


def dyck_member(s: bytes, max_depth=3) -> bool:
    stack = []
    for c in s:
        if c in b"{[":
            stack.append(c)
            if len(stack) > max_depth:
                return False
        elif c in b"}]":
            if not stack or stack[-1] != {ord("}"): ord("{"), ord("]"): ord("[")}[c]:
                return False
            stack.pop()
        else:
            ctx = stack[-1] if stack else None
            want = {None: ord("c"), ord("{"): ord("a"), ord("["): ord("b")}[ctx]
            if c != want:
                return False
    return not stack


def dyck2_member(s: bytes, max_depth=3) -> bool:
    stack = []
    for c in s:
        if c in b"{[":
            stack.append(c)
            if len(stack) > max_depth:
                return False
        elif c in b"}]":
            if not stack or stack.pop() != {ord("}"): ord("{"), ord("]"): ord("[")}[c]:
                return False
        elif c != ord("a"):
            return False
    return not stack


INT_RE = re.compile(rb"-?(0|[1-9][0-9]*)")


def int_member(s: bytes) -> bool:
    return INT_RE.fullmatch(s) is not None


def language(alphabet: bytes, N: int, member):
    members = set()
    for L in range(N + 1):
        for tup in itertools.product(alphabet, repeat=L):
            s = bytes(tup)
            if member(s):
                members.add(s)
    viable = set()
    for m in members:
        for i in range(len(m) + 1):
            viable.add(m[:i])
    return members, viable


def open_count(p: bytes, opens=b"([{") -> int:
    d = 0
    for c in p:
        if c in opens:
            d += 1
        elif c in b")]}":
            d = max(0, d - 1)
    return d


def brute_force_check(oracle, automaton, alphabet, N, member, completion_bound, max_prefix, max_tok):
    members, viable = language(alphabet, N, member)
    vocab = synth.all_strings_vocab(alphabet, max_tok)
    toks = vocab.tokens()
    P = oracle.Problem.from_parts(automaton, vocab)
    prefixes = sorted(p for p in viable if len(p) <= max_prefix)
    # a few rejected prefixes as well: their walk must fail
    rejected = [bytes(t) for L in range(1, 4) for t in itertools.product(alphabet, repeat=L)
                if bytes(t) not in viable][:50]
    for u in rejected:
        assert walk_prefix(oracle, automaton, u) is None, u
    cfgs = [walk_prefix(oracle, automaton, u) for u in prefixes]
    assert all(c is not None for c in cfgs), [u for u, c in zip(prefixes, cfgs) if c is None][:5]
    states = np.array([c[0] for c in cfgs], np.int32)
    stacks = np.array([c[1] for c in cfgs], np.uint64)
    mask, nxt, bad = P.step_mask(states, stacks, want_next=True)
    assert bad == 0
    compared = 0
    for i, u in enumerate(prefixes):
        bits = oracle.bits_of(mask[i], vocab.n_tokens)
        for t, tok in enumerate(toks):
            if t == vocab.eos_id:
                assert bits[t] == (u in members), (u, "EOS")
                compared += 1
                continue
            p = u + tok
            if p in viable:
                assert bits[t], (u, tok)
                compared += 1
            elif len(p) + completion_bound(p) <= N:
                assert not bits[t], (u, tok)
                compared += 1
    return compared


def test_brute_force_fig3_expression(oracle_lib):
    n = brute_force_check(oracle_lib, synth.fig3_expr_pda(), b"01(+) ", 7, expr_member,
                          lambda p: open_count(p) + 1, max_prefix=4, max_tok=3)
    assert n > 5000


def test_brute_force_fig3_expression_depth_bound(oracle_lib):
    # max_depth = 2: a third open parenthesis must be rejected (bounded stack)
    n = brute_force_check(oracle_lib, synth.fig3_expr_pda(max_depth=2), b"1(+) ", 7,
                          lambda s: expr_member(s, max_depth=2), lambda p: open_count(p) + 1, max_prefix=4,
                          max_tok=3)
    assert n > 2000


def test_brute_force_dyck_with_context(oracle_lib):
    n = brute_force_check(oracle_lib, synth.dyck_ctx_pda(max_depth=3), b"{}[]abc", 7, dyck_member,
                          lambda p: open_count(p), max_prefix=4, max_tok=3)
    assert n > 20000


def test_brute_force_dyck2_top_of_stack(oracle_lib):
    n = brute_force_check(oracle_lib, synth.dyck2_pda(max_depth=3), b"{}[]a", 8, dyck2_member,
                          lambda p: open_count(p), max_prefix=5, max_tok=3)
    assert n > 20000


def test_brute_force_int_regex(oracle_lib):
    n = brute_force_check(oracle_lib, synth.int_regex_dfa(), b"-0123", 7, int_member, lambda p: 1,
                          max_prefix=4, max_tok=3)
    assert n > 1000


# --------------------------------------------------------------------------
# single-byte tokens and invariants on the workloads
# --------------------------------------------------------------------------
@pytest.mark.parametrize("config", [1, 2])
def test_single_byte_tokens_equal_live_out_bytes(oracle_lib, config):
    w = synth.workload(config)
    a, v = w.automaton, w.vocab
    toks = v.tokens()
    single = {tok[0]: t for t, tok in enumerate(toks) if len(tok) == 1}
    P = oracle_lib.Problem.from_workload(w)
    qs = np.nonzero(a.live)[0].astype(np.int32)
    mask, _, _ = P.step_mask(qs)
    for i, q in enumerate(qs):
        bits = oracle_lib.bits_of(mask[i], v.n_tokens)
        for c, t in single.items():
            assert bits[t] == bool(a.live[a.delta[q, c]]), (q, c)


@pytest.mark.parametrize("config", [2, 3, 5])
def test_next_state_invariants(oracle_lib, config):
    w = synth.workload(config)
    a = w.automaton
    P = oracle_lib.Problem.from_workload(w)
    states, stacks = w.initial_configs(batch=4)
    mask, nxt, bad = P.step_mask(states, stacks, want_next=True)
    assert bad == 0
    for i in range(len(states)):
        bits = oracle_lib.bits_of(mask[i], w.vocab.n_tokens)
        assert np.all(nxt[i][~bits] == 0)
        assert np.all(nxt[i][bits] != 0)
        assert np.all(a.live[nxt[i][bits]] == 1)
        assert bits.any()


@pytest.mark.parametrize("config", [3, 5])
def test_next_state_composition(oracle_lib, config):
    """next(q, t1.t2) == next(next(q, t1), t2) and allowed(t1.t2) iff both steps are."""
    w = synth.workload(config)
    rng = np.random.default_rng(7)
    toks = w.vocab.tokens()
    pairs = [(toks[i], toks[j]) for i, j in rng.integers(0, w.vocab.n_tokens - 1, size=(400, 2))]
    cat = [a + b for a, b in pairs]
    vocab = synth.Vocab.from_tokens([p[0] for p in pairs] + [p[1] for p in pairs] + cat)
    P = oracle_lib.Problem.from_parts(w.automaton, vocab)
    states, stacks = w.initial_configs(batch=6)
    n = len(pairs)
    for s, st in zip(states, stacks):
        for k in range(n):
            r12, s12, w12 = P.check(s, st, 2 * n + k)
            r1, s1, w1 = P.check(s, st, k)
            if r1 != 1:
                assert r12 == 0
                continue
            r2, s2, w2 = P.check(s1, w1, n + k)
            assert r12 == r2
            if r12 == 1:
                assert (s12, w12) == (s2, w2)


def test_stack_depth_bounds(oracle_lib):
    w = synth.workload(5)
    P = oracle_lib.Problem.from_workload(w)
    toks = w.vocab.tokens()
    states, stacks = w.initial_configs(batch=8)
    rng = np.random.default_rng(3)
    ids = rng.integers(0, w.vocab.n_tokens - 1, size=3000)
    for s, st in zip(states, stacks):
        before = synth.unpack_stack(int(st))
        for t in ids:
            r, s2, w2 = P.check(s, st, int(t))
            if r != 1:
                continue
            after = synth.unpack_stack(w2)
            L = len(toks[t])
            assert 0 <= len(after) <= 32
            assert abs(len(after) - len(before)) <= L
            keep = max(0, len(before) - L)
            assert after[:keep] == before[:keep]


# --------------------------------------------------------------------------
# masked logits (Alg. 1: v' = m (.) v, decode = argmax; log-softmax)
# --------------------------------------------------------------------------
def pack_bits(bits: np.ndarray) -> np.ndarray:
    V = bits.shape[-1]
    W = (V + 31) // 32
    padded = np.zeros(bits.shape[:-1] + (W * 32,), dtype=np.uint8)
    padded[..., :V] = bits
    return np.packbits(padded, axis=-1, bitorder="little").view("<u4")


def test_logits_uniform_and_single(oracle_lib):
    V = 77
    x = np.full((3, V), 0.75, np.float32)
    bits = np.zeros((3, V), bool)
    bits[0, [3, 9, 40, 76]] = True          # 4 allowed -> logprob = -log 4
    bits[1, 50] = True                      # one allowed -> logprob 0
    # row 2: nothing allowed
    arg, lse, lp = oracle_lib.mask_logits(x, pack_bits(bits), want_logprobs=True)
    assert arg.tolist() == [3, 50, -1]
    assert math.isclose(lse[0], 0.75 + math.log(4), abs_tol=1e-12)
    assert np.allclose(lp[0][bits[0]], -math.log(4), atol=1e-12)
    assert np.all(np.isneginf(lp[0][~bits[0]]))
    assert lp[1, 50] == 0.0 and lse[1] == 0.75
    assert np.isneginf(lse[2]) and np.all(np.isneginf(lp[2]))


def test_logits_ties_lowest_index_and_mask_wins(oracle_lib):
    V = 100
    x = np.zeros((1, V), np.float32)
    x[0, [10, 20, 30]] = 5.0
    x[0, 5] = 9.0                            # larger but masked
    bits = np.ones((1, V), bool)
    bits[0, 5] = False
    bits[0, 10] = False
    arg, _, _ = oracle_lib.mask_logits(x, pack_bits(bits))
    assert arg[0] == 20


def test_logits_against_scipy_and_normalisation(oracle_lib):
    scipy_special = pytest.importorskip("scipy.special")
    rng = np.random.default_rng(11)
    B, V = 5, 1000
    x32 = (rng.standard_normal((B, V)) * 3).astype(np.float32)
    xb = synth.f32_to_bf16_bits(x32)
    xv = synth.bf16_bits_to_f32(xb).astype(np.float64)
    bits = rng.random((B, V)) < 0.3
    arg, lse, lp = oracle_lib.mask_logits(xb, pack_bits(bits), want_logprobs=True)
    for b in range(B):
        ref = scipy_special.logsumexp(xv[b][bits[b]])
        assert abs(lse[b] - ref) < 1e-9
        assert abs(np.exp(lp[b][bits[b]]).sum() - 1.0) < 1e-9
        masked = np.where(bits[b], xv[b], -np.inf)
        assert arg[b] == int(np.argmax(masked))      # numpy returns the first maximum


def test_bf16_values_are_exact(oracle_lib):
    bits = np.array([[0x3F80, 0xC000, 0x3F81, 0x0000, 0x4049]], np.uint16)   # 1, -2, 1.0078125, 0, 3.140625
    m = pack_bits(np.array([[True, True, True, True, True]]))
    arg, lse, lp = oracle_lib.mask_logits(bits, m, want_logprobs=True)
    assert arg[0] == 4
    ref = math.log(math.exp(1) + math.exp(-2) + math.exp(1.0078125) + 1 + math.exp(3.140625))
    assert abs(lse[0] - ref) < 1e-12


def test_logits_row_stride(oracle_lib):
    rng = np.random.default_rng(5)
    x = rng.standard_normal((3, 48)).astype(np.float32)
    bits = rng.random((3, 40)) < 0.5
    a1, l1, p1 = oracle_lib.mask_logits(x, pack_bits(bits), n_tokens=40, want_logprobs=True)
    a2, l2, p2 = oracle_lib.mask_logits(np.ascontiguousarray(x[:, :40]), pack_bits(bits), want_logprobs=True)
    assert (a1 == a2).all() and np.allclose(l1, l2) and np.allclose(p1, p2)


# --------------------------------------------------------------------------
# edge shapes and invalid configurations
# --------------------------------------------------------------------------
def test_edge_shapes(oracle_lib):
    a = synth.int_regex_dfa()
    toks = [b"1", b"-", b"0", b"1" * 32, b"12", b"-0", b"00"] + [bytes([c]) for c in b"abcdefghijklmnopqrstuvwxy"]
    toks.append(b"")                                                   # an empty token that is not EOS
    v = synth.Vocab.from_tokens(toks, eos_id=-1)                       # no EOS, V = 33
    P = oracle_lib.Problem.from_parts(a, v)
    mask, nxt, bad = P.step_mask(np.array([a.start, 0, 99, -1], np.int32), want_next=True)
    assert bad == 2                                                    # 99 and -1 are out of range
    assert v.n_tokens == 33 and mask.shape == (4, 2)
    assert (mask[0, 1] >> 1) == 0                                      # pad bits above V are zero
    bits = oracle_lib.bits_of(mask[0], 33)
    assert bits[:7].tolist() == [True, True, True, True, True, True, False]
    assert not bits[7:].any()
    assert (mask[1:] == 0).all() and (nxt[1:] == 0).all()              # dead and invalid rows


def test_invalid_stacks_and_depth_limit(oracle_lib):
    a = synth.dyck_ctx_pda(max_depth=32)
    v = synth.Vocab.from_tokens([b"{", b"}", b"a", b"c", b""], eos_id=4)
    P = oracle_lib.Problem.from_parts(a, v)
    full = synth.pack_stack([0] * 32)
    states = np.array([2, 2, 1, 1, 1, 2], np.int32)
    stacks = np.array([full, (33 << 32), (1 << 32) | 2, (1 << 40), 0, synth.pack_stack([0])], np.uint64)
    mask, _, bad = P.step_mask(states, stacks)
    assert bad == 3                         # depth 33 > max, a bit above the depth, bits >= 40 set
    row = lambda i: oracle_lib.bits_of(mask[i], v.n_tokens).tolist()
    assert row(0) == [False, True, True, False, False]     # depth 32: '{' would overflow
    assert row(4) == [True, False, False, True, True]      # top level: '{', 'c', EOS
    assert row(5) == [True, True, True, False, False]      # inside one '{'


def test_advance_rules(oracle_lib):
    a = synth.fig3_expr_pda()
    v = synth.fig3_vocab()
    P = oracle_lib.Problem.from_parts(a, v)
    toks = v.tokens()
    states = np.array([1, 1, 2, 4, 1, 3, 2], np.int32)
    stacks = np.array([0, 0, synth.pack_stack([0]), 0, 0, 0, synth.pack_stack([0, 0])], np.uint64)
    tokens = np.array([toks.index(b"("), toks.index(b")"), -1, v.eos_id, 99, toks.index(b"+"),
                       toks.index(b")")], np.int32)
    so, wo, bad = P.advance(states, stacks, tokens, a.start)
    assert bad == 1                                        # token id 99 >= V
    assert so.tolist() == [1, 0, a.start, a.start, 0, 1, 4]
    assert wo.tolist() == [synth.pack_stack([0]), 0, 0, 0, 0, 0, synth.pack_stack([0])]
