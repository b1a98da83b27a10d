"""Seeded synthetic workloads: vocabularies, automata, batch states and logits.

This module only BUILDS INPUTS.  It holds none of the method's arithmetic (no
token walk, no mask, no log-softmax): the automata are written down directly
as transition tables, the vocabularies are random byte strings, and the batch
configurations come from a random walk that this module takes over the
automaton it has just built (that is how a reachable (state, stack) pair is
produced for the pushdown workload).  Both the CPU oracle and the CUDA library
consume what it returns.

Shapes follow the paper's workloads (JSON-like grammars over a BPE vocabulary,
Sec. 4 and App. C); the vocabularies and grammars of the paper are not
available, so these seeded stand-ins replace them:

  config 1  16-state DFA for a one-level `{ "key": value, ... }` language,
            V = 1024 over the 42-byte alphabet [0-9a-z{}":, ], batch 1, fp32.
  config 2  200-state DFA: objects over 8 fixed keys (a key trie), values
            "[^"\\]*" or -?[0-9]+, V = 32000, batch 32, bf16 N(0, 2).
  config 3  random sparse DFA, Q = 5000, 32 byte classes, 8 live classes per
            state, V = 128256, batch 256, bf16 N(0, 3).
  config 4  the config-3 generator with Q = 20000 (state x token precompute).
  config 5  300-state JSON lexer (after the paper's basic JSON grammar,
            App. C) with a {/[ bracket stack of depth <= 32, V = 152064,
            batch 128, bf16 N(0, 3), log-probs requested.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

RULE_PUSH = 1
RULE_POP = 2

# One stack rule (state, byte) -> PUSH sym | POP sym; the three targets are
# used by POP only (next state chosen by the symbol revealed after the pop).
RULE_DTYPE = np.dtype([
    ("state", "<i4"), ("byte", "u1"), ("kind", "u1"), ("sym", "u1"), ("pad", "u1"),
    ("next_if_empty", "<i4"), ("next_if_top0", "<i4"), ("next_if_top1", "<i4"),
])

WS_JSON = b" \t\n"
WS_KV = b" \t\n\r"
DIGITS = b"0123456789"
LOWER = b"abcdefghijklmnopqrstuvwxyz"
HEX = b"0123456789abcdefABCDEF"


# --------------------------------------------------------------------------
# containers
# --------------------------------------------------------------------------
@dataclasses.dataclass
class Vocab:
    data: np.ndarray      # uint8, all token byte strings concatenated
    offsets: np.ndarray   # int64 [V+1]
    eos_id: int           # -1: no EOS token

    @property
    def n_tokens(self) -> int:
        return int(self.offsets.shape[0] - 1)

    def token(self, t: int) -> bytes:
        return bytes(self.data[self.offsets[t]:self.offsets[t + 1]])

    def tokens(self) -> List[bytes]:
        d = self.data.tobytes()
        o = self.offsets
        return [d[o[i]:o[i + 1]] for i in range(self.n_tokens)]

    @staticmethod
    def from_tokens(tokens: Sequence[bytes], eos_id: int = -1) -> "Vocab":
        lens = np.array([len(t) for t in tokens], dtype=np.int64)
        offsets = np.zeros(len(tokens) + 1, dtype=np.int64)
        np.cumsum(lens, out=offsets[1:])
        data = np.frombuffer(b"".join(tokens), dtype=np.uint8).copy()
        if data.size == 0:
            data = np.zeros(1, dtype=np.uint8)
        return Vocab(data=data, offsets=offsets, eos_id=eos_id)


@dataclasses.dataclass
class Automaton:
    delta: np.ndarray              # int32 [Q][256]; state 0 is the dead state
    live: np.ndarray               # uint8 [Q]: state can still reach acceptance
    accepting: np.ndarray          # uint8 [Q]
    start: int
    rules: Optional[np.ndarray]    # RULE_DTYPE records, or None for a plain DFA
    max_depth: int                 # bracket-stack bound (0 for a plain DFA)
    name: str = ""

    @property
    def n_states(self) -> int:
        return int(self.delta.shape[0])

    @property
    def n_rules(self) -> int:
        return 0 if self.rules is None else int(self.rules.shape[0])


@dataclasses.dataclass
class Workload:
    config: int
    name: str
    automaton: Automaton
    vocab: Vocab
    batch: int
    steps: int
    logits_dtype: str          # "f32" or "bf16"
    logits_sigma: float
    want_logprobs: bool
    description: str

    def seed(self, *parts: int) -> np.random.Generator:
        return np.random.default_rng([1000 + self.config, *parts])

    def initial_configs(self, batch: Optional[int] = None, part: int = 2) -> Tuple[np.ndarray, np.ndarray]:
        """(states int32 [B], stacks uint64 [B]) drawn from this workload's recipe."""
        b = self.batch if batch is None else batch
        rng = self.seed(part)
        a = self.automaton
        if a.rules is None:
            live_ids = np.nonzero(a.live)[0]
            states = rng.choice(live_ids, size=b).astype(np.int32)
            return states, np.zeros(b, dtype=np.uint64)
        states = np.zeros(b, dtype=np.int32)
        stacks = np.zeros(b, dtype=np.uint64)
        for i in range(b):
            target = int(rng.integers(0, a.max_depth + 1))
            s, stk = random_pda_walk(a, rng, target)
            states[i] = s
            stacks[i] = pack_stack(stk)
        return states, stacks

    def logits(self, step: int, batch: Optional[int] = None) -> np.ndarray:
        """Logits for one decode step: float32 [B][V] or bf16 bits uint16 [B][V]."""
        b = self.batch if batch is None else batch
        return make_logits(self.seed(3, step), b, self.vocab.n_tokens, self.logits_sigma, self.logits_dtype)


# --------------------------------------------------------------------------
# small helpers
# --------------------------------------------------------------------------
def pack_stack(symbols: Sequence[int]) -> int:
    """Boundary encoding of a bracket stack: bits 0..31 hold the symbols with
    the top at bit 0, bits 32..39 hold the depth."""
    bits = 0
    for sym in symbols:           # bottom first
        bits = (bits << 1) | (sym & 1)
    return (len(symbols) << 32) | bits


def unpack_stack(word: int) -> List[int]:
    depth = (int(word) >> 32) & 0xFF
    bits = int(word) & 0xFFFFFFFF
    return [(bits >> (depth - 1 - i)) & 1 for i in range(depth)]


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even float32 -> bfloat16, returned as raw uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (b.astype(np.uint32) << 16).view(np.float32)


def make_logits(rng: np.random.Generator, batch: int, n_tokens: int, sigma: float, dtype: str) -> np.ndarray:
    x = rng.standard_normal((batch, n_tokens), dtype=np.float32) * np.float32(sigma)
    if dtype == "f32":
        return x
    if dtype == "bf16":
        return f32_to_bf16_bits(x)
    raise ValueError(dtype)


class _Builder:
    """Incremental DFA / bracket-PDA table writer."""

    def __init__(self):
        self.rows: List[np.ndarray] = [np.zeros(256, dtype=np.int32)]   # state 0: dead
        self.names: List[str] = ["dead"]
        self.accept: List[int] = [0]
        self.rules: Dict[Tuple[int, int], tuple] = {}

    def state(self, name: str, accepting: bool = False) -> int:
        self.rows.append(np.zeros(256, dtype=np.int32))
        self.names.append(name)
        self.accept.append(1 if accepting else 0)
        return len(self.rows) - 1

    def edge(self, s: int, chars, t: int) -> None:
        for c in (chars if isinstance(chars, (bytes, bytearray, list, range)) else [chars]):
            c = c if isinstance(c, int) else ord(c)
            self.rows[s][c] = t

    def push(self, s: int, char: bytes, sym: int, t: int) -> None:
        c = char[0]
        self.rows[s][c] = t
        self.rules[(s, c)] = (RULE_PUSH, sym, 0, 0, 0)

    def pop(self, s: int, char: bytes, sym: int, ret: Tuple[int, int, int]) -> None:
        c = char[0]
        self.rows[s][c] = 0        # the target comes from the revealed stack top
        self.rules[(s, c)] = (RULE_POP, sym) + tuple(ret)

    def build(self, start: int, max_depth: int, name: str, live: Optional[np.ndarray] = None) -> Automaton:
        delta = np.stack(self.rows).astype(np.int32)
        acc = np.array(self.accept, dtype=np.uint8)
        if live is None:
            live = np.ones(delta.shape[0], dtype=np.uint8)
            live[0] = 0
        rules = None
        if self.rules:
            rules = np.zeros(len(self.rules), dtype=RULE_DTYPE)
            for i, ((s, c), r) in enumerate(sorted(self.rules.items())):
                rules[i] = (s, c, r[0], r[1], 0, r[2], r[3], r[4])
        return Automaton(delta=delta, live=live, accepting=acc, start=start,
                         rules=rules, max_depth=max_depth if rules is not None else 0, name=name)


def random_pda_walk(a: Automaton, rng: np.random.Generator, target_depth: int,
                    max_steps: int = 4000) -> Tuple[int, List[int]]:
    """Random legal byte walk from (start, empty) until the stack depth equals
    `target_depth`, then a few more depth-preserving bytes.  Outcomes are
    grouped by (kind, next state) and picked uniformly, so the walk visits many
    different lexer states instead of staying inside strings."""
    rule_at = {}
    for r in a.rules:
        rule_at[(int(r["state"]), int(r["byte"]))] = r
    s, stk = a.start, []
    extra = int(rng.integers(0, 13))
    for _ in range(max_steps):
        if len(stk) == target_depth:
            if extra == 0:
                break
            extra -= 1
        groups: Dict[tuple, List[int]] = {}
        for c in range(256):
            r = rule_at.get((s, c))
            if r is None:
                t = int(a.delta[s, c])
                if t != 0 and a.live[t]:
                    groups.setdefault(("step", t), []).append(c)
            elif r["kind"] == RULE_PUSH:
                if len(stk) < min(target_depth, a.max_depth):
                    t = int(a.delta[s, c])
                    if t != 0 and a.live[t]:
                        groups.setdefault(("push", t, int(r["sym"])), []).append(c)
            # never pop: the walk only climbs to its target depth
        if not groups:
            break
        keys = list(groups.keys())
        push_keys = [k for k in keys if k[0] == "push"]
        if push_keys and len(stk) < target_depth and rng.random() < 0.5:
            key = push_keys[int(rng.integers(0, len(push_keys)))]
        else:
            step_keys = [k for k in keys if k[0] == "step"] or keys
            key = step_keys[int(rng.integers(0, len(step_keys)))]
        if key[0] == "push":
            stk.append(key[2])
        s = key[1]
    return s, stk


# --------------------------------------------------------------------------
# vocabularies
# --------------------------------------------------------------------------
def _mixed_bytes(rng: np.random.Generator, n: int) -> np.ndarray:
    """95 % printable 0x20..0x7E, 5 % high bytes 0x80..0xFF."""
    hi = rng.random(n) < 0.05
    out = rng.integers(0x20, 0x7F, size=n).astype(np.uint8)
    out[hi] = rng.integers(0x80, 0x100, size=int(hi.sum())).astype(np.uint8)
    return out


def random_vocab(rng: np.random.Generator, n_tokens: int, singles: bytes, length_sampler, byte_sampler,
                 eos: bool = True) -> Vocab:
    """Ids 0..len(singles)-1 are the single bytes `singles`; the rest are unique
    random strings (duplicates and collisions with the singles are resampled);
    the last id is the zero-length EOS token when `eos`."""
    tokens: List[bytes] = [bytes([c]) for c in singles]
    seen = set(tokens)
    need = n_tokens - len(tokens) - (1 if eos else 0)
    while need > 0:
        m = max(1024, int(need * 1.3))
        lens = length_sampler(rng, m)
        data = byte_sampler(rng, int(lens.sum())).tobytes()
        pos = 0
        for L in lens.tolist():
            s = data[pos:pos + L]
            pos += L
            if s in seen:
                continue
            seen.add(s)
            tokens.append(s)
            need -= 1
            if need == 0:
                break
    if eos:
        tokens.append(b"")
    return Vocab.from_tokens(tokens, eos_id=(len(tokens) - 1) if eos else -1)


def geometric_lengths(mean: float, max_len: int):
    p = 1.0 / mean

    def sample(rng, m):
        out = rng.geometric(p, size=m)
        bad = out > max_len
        while bad.any():                       # truncation by resampling
            out[bad] = rng.geometric(p, size=int(bad.sum()))
            bad = out > max_len
        return out.astype(np.int64)
    return sample


# --------------------------------------------------------------------------
# config 1: 16-state key/value DFA, alphabet [0-9a-z{}":, ]
# --------------------------------------------------------------------------
CFG1_ALPHABET = b'0123456789abcdefghijklmnopqrstuvwxyz{}":, '


def kv16_dfa() -> Automaton:
    b = _Builder()
    START = b.state("start")
    OPEN = b.state("open")
    KQ = b.state("key_quote")
    KEY = b.state("key")
    KEND = b.state("key_end")
    COLON = b.state("colon")
    ZERO = b.state("val_zero")
    INT = b.state("val_int")
    IDENT = b.state("val_ident")
    AFTERV = b.state("after_value")
    CLOSED = b.state("closed", accepting=True)
    COMMA = b.state("comma")
    VSO = b.state("vstr_open")
    VSTR = b.state("vstr")
    VSE = b.state("vstr_end")
    alnum = LOWER + DIGITS
    b.edge(START, b" ", START); b.edge(START, b"{", OPEN)
    b.edge(OPEN, b" ", OPEN); b.edge(OPEN, b'"', KQ); b.edge(OPEN, b"}", CLOSED)
    b.edge(KQ, LOWER, KEY)
    b.edge(KEY, alnum, KEY); b.edge(KEY, b'"', KEND)
    b.edge(KEND, b" ", KEND); b.edge(KEND, b":", COLON)
    b.edge(COLON, b" ", COLON); b.edge(COLON, b"0", ZERO); b.edge(COLON, b"123456789", INT)
    b.edge(COLON, LOWER, IDENT); b.edge(COLON, b'"', VSO)
    for v in (ZERO, INT, IDENT, AFTERV, VSE):
        b.edge(v, b" ", AFTERV); b.edge(v, b",", COMMA); b.edge(v, b"}", CLOSED)
    b.edge(INT, DIGITS, INT)
    b.edge(IDENT, alnum, IDENT)
    b.edge(CLOSED, b" ", CLOSED)
    b.edge(COMMA, b" ", COMMA); b.edge(COMMA, b'"', KQ)
    b.edge(VSO, alnum + b" ", VSTR); b.edge(VSO, b'"', VSE)
    b.edge(VSTR, alnum + b" ", VSTR); b.edge(VSTR, b'"', VSE)
    a = b.build(START, 0, "kv16")
    assert a.n_states == 16
    return a


# --------------------------------------------------------------------------
# config 2: ~200-state DFA over 8 fixed keys
# --------------------------------------------------------------------------
def _distinct_first_keys(rng: np.random.Generator, n_keys: int, total_len: int, lo: int, hi: int) -> List[bytes]:
    """n_keys random lowercase keys with pairwise distinct first letters whose
    lengths sum to total_len (so the key trie has exactly total_len non-root nodes)."""
    assert n_keys <= 26 and lo * n_keys <= total_len <= hi * n_keys
    lens = np.full(n_keys, total_len // n_keys)
    lens[: total_len - lens.sum()] += 1
    for _ in range(4 * n_keys):                  # random but sum-preserving jitter
        i, j = rng.integers(0, n_keys, size=2)
        d = int(rng.integers(0, 4))
        if lens[i] - d >= lo and lens[j] + d <= hi:
            lens[i] -= d
            lens[j] += d
    firsts = rng.permutation(26)[:n_keys]
    keys = []
    for k in range(n_keys):
        body = rng.integers(0, 26, size=int(lens[k]) - 1)
        keys.append(bytes([LOWER[firsts[k]]] + [LOWER[x] for x in body]))
    return keys


def _add_trie(b: _Builder, root: int, keys: Sequence[bytes], on_full, on_other=None) -> int:
    """Adds one state per non-root trie node; on_full(node) adds the edges of a
    node that spells a whole key; on_other(node) the edges every node gets."""
    nodes = {b"": root}
    count = 0
    for key in keys:
        for i in range(1, len(key) + 1):
            p = key[:i]
            if p not in nodes:
                nodes[p] = b.state("key:" + p.decode())
                count += 1
    for p, s in nodes.items():
        if on_other is not None:
            on_other(s)
    for p, s in nodes.items():
        for q, t in nodes.items():
            if len(q) == len(p) + 1 and q[:-1] == p:
                b.edge(s, q[-1], t)
    for key in keys:
        on_full(nodes[key])
    return count


def kv200_dfa(rng: np.random.Generator) -> Tuple[Automaton, List[bytes]]:
    b = _Builder()
    START = b.state("start")
    OPEN = b.state("open")
    KROOT = b.state("key_root")
    KEND = b.state("key_end")
    COLON = b.state("colon")
    VSTR = b.state("vstr")
    NEG = b.state("neg")
    VINT = b.state("vint")
    AFTERV = b.state("after_value")
    COMMA = b.state("comma")
    CLOSED = b.state("closed", accepting=True)
    n_fixed = len(b.rows)          # 12 including the dead state
    keys = _distinct_first_keys(rng, 8, 200 - n_fixed, 12, 36)
    b.edge(START, WS_KV, START); b.edge(START, b"{", OPEN)
    b.edge(OPEN, WS_KV, OPEN); b.edge(OPEN, b'"', KROOT); b.edge(OPEN, b"}", CLOSED)
    _add_trie(b, KROOT, keys, on_full=lambda s: b.edge(s, b'"', KEND))
    b.edge(KEND, WS_KV, KEND); b.edge(KEND, b":", COLON)
    b.edge(COLON, WS_KV, COLON); b.edge(COLON, b'"', VSTR); b.edge(COLON, b"-", NEG); b.edge(COLON, DIGITS, VINT)
    b.edge(VSTR, [c for c in range(256) if c not in (0x22, 0x5C)], VSTR); b.edge(VSTR, b'"', AFTERV)
    b.edge(NEG, DIGITS, VINT)
    b.edge(VINT, DIGITS, VINT)
    for v in (VINT, AFTERV):
        b.edge(v, WS_KV, AFTERV); b.edge(v, b",", COMMA); b.edge(v, b"}", CLOSED)
    b.edge(COMMA, WS_KV, COMMA); b.edge(COMMA, b'"', KROOT)
    b.edge(CLOSED, WS_KV, CLOSED)
    a = b.build(START, 0, "kv200")
    assert a.n_states == 200, a.n_states
    return a, keys


# --------------------------------------------------------------------------
# configs 3/4: random sparse DFA
# --------------------------------------------------------------------------
def random_sparse_dfa(rng: np.random.Generator, n_states: int, n_classes: int = 32, live_per_state: int = 8,
                      accept_frac: float = 0.1) -> Automaton:
    """Bytes are split into n_classes random classes of equal size; every state
    1..Q-1 has live_per_state live classes with random targets; states
    1..Q*accept_frac are accepting and every other state i has one live edge to
    a state < i, so all states are co-reachable to acceptance by induction."""
    Q = n_states
    n_acc = int(Q * accept_frac)
    cls_of_byte = np.empty(256, dtype=np.int64)
    cls_of_byte[rng.permutation(256)] = np.arange(256) * n_classes // 256
    order = np.argsort(rng.random((Q, n_classes)), axis=1)[:, :live_per_state]
    targets = rng.integers(1, Q, size=(Q, live_per_state))
    down = (rng.random(Q) * np.maximum(np.arange(Q) - 1, 1)).astype(np.int64) + 1   # uniform in [1, q-1]
    non_acc = np.arange(Q) > n_acc
    targets[non_acc, 0] = down[non_acc]
    dc = np.zeros((Q, n_classes), dtype=np.int32)
    np.put_along_axis(dc, order, targets.astype(np.int32), axis=1)
    dc[0, :] = 0
    delta = np.ascontiguousarray(dc[:, cls_of_byte])
    live = np.ones(Q, dtype=np.uint8)
    live[0] = 0
    acc = np.zeros(Q, dtype=np.uint8)
    acc[1:n_acc + 1] = 1
    return Automaton(delta=delta, live=live, accepting=acc, start=1, rules=None, max_depth=0,
                     name=f"sparse{Q}")


# --------------------------------------------------------------------------
# config 5: JSON lexer with bracket stack (after the paper's JSON grammar)
# --------------------------------------------------------------------------
def json_pda(rng: np.random.Generator, n_states: int = 300, max_depth: int = 32) -> Tuple[Automaton, List[bytes]]:
    """Root is an object; values are object | array | string | number |
    true/false/null; ws is [ \\t\\n]; strings are [^"\\\\] or escapes
    (\\["\\\\/bfnrt] or \\u + 4 hex digits).  '{' pushes 0 and '[' pushes 1;
    '}' / ']' pop their own symbol and go to the after-value state of the
    container that the pop reveals (or to the final state at depth 0).  Keys
    are any string; a trie of fixed keys tracks well-known keys (states that
    behave like the generic key-string state) and pads the lexer to n_states."""
    b = _Builder()
    START = b.state("top_start")
    DONE = b.state("top_done", accepting=True)
    OBJ_OPEN = b.state("obj_open")
    OBJ_COMMA = b.state("obj_comma")
    KROOT = b.state("key_root")
    KSTR = b.state("key_str")
    KESC = b.state("key_esc")
    KU = [b.state(f"key_u{i}") for i in range(4)]
    KEND = b.state("key_end")
    OBJ_COLON = b.state("obj_colon")
    ARR_OPEN = b.state("arr_open")
    ARR_COMMA = b.state("arr_comma")
    ctx = {}
    for c in ("obj", "arr"):
        d = {}
        for nm in ("str", "esc", "u0", "u1", "u2", "u3",
                   "minus", "zero", "int", "dot", "frac", "e", "esign", "exp",
                   "t1", "t2", "t3", "f1", "f2", "f3", "f4", "n1", "n2", "n3", "av"):
            d[nm] = b.state(f"{c}_{nm}")
        ctx[c] = d
    n_fixed = len(b.rows)
    content = [c for c in range(0x100) if c not in (0x22, 0x5C)]
    ret = (DONE, ctx["obj"]["av"], ctx["arr"]["av"])

    def follow(s, c):
        """Edges that may follow a complete value in container c."""
        b.edge(s, WS_JSON, ctx[c]["av"])
        if c == "obj":
            b.edge(s, b",", OBJ_COMMA)
            b.pop(s, b"}", 0, ret)
        else:
            b.edge(s, b",", ARR_COMMA)
            b.pop(s, b"]", 1, ret)

    def value_start(s, c):
        d = ctx[c]
        b.edge(s, b'"', d["str"]); b.edge(s, b"-", d["minus"]); b.edge(s, b"0", d["zero"])
        b.edge(s, b"123456789", d["int"])
        b.edge(s, b"t", d["t1"]); b.edge(s, b"f", d["f1"]); b.edge(s, b"n", d["n1"])
        b.push(s, b"{", 0, OBJ_OPEN)
        b.push(s, b"[", 1, ARR_OPEN)

    def string_body(s_str, s_esc, us, s_close):
        b.edge(s_str, content, s_str); b.edge(s_str, b'"', s_close); b.edge(s_str, b"\\", s_esc)
        b.edge(s_esc, b'"\\/bfnrt', s_str); b.edge(s_esc, b"u", us[0])
        for i in range(3):
            b.edge(us[i], HEX, us[i + 1])
        b.edge(us[3], HEX, s_str)

    b.edge(START, WS_JSON, START); b.push(START, b"{", 0, OBJ_OPEN)
    b.edge(DONE, WS_JSON, DONE)
    b.edge(OBJ_OPEN, WS_JSON, OBJ_OPEN); b.edge(OBJ_OPEN, b'"', KROOT); b.pop(OBJ_OPEN, b"}", 0, ret)
    b.edge(OBJ_COMMA, WS_JSON, OBJ_COMMA); b.edge(OBJ_COMMA, b'"', KROOT)
    string_body(KSTR, KESC, KU, KEND)
    b.edge(KEND, WS_JSON, KEND); b.edge(KEND, b":", OBJ_COLON)
    b.edge(OBJ_COLON, WS_JSON, OBJ_COLON); value_start(OBJ_COLON, "obj")
    b.edge(ARR_OPEN, WS_JSON, ARR_OPEN); value_start(ARR_OPEN, "arr"); b.pop(ARR_OPEN, b"]", 1, ret)
    b.edge(ARR_COMMA, WS_JSON, ARR_COMMA); value_start(ARR_COMMA, "arr")
    for c, d in ctx.items():
        string_body(d["str"], d["esc"], [d["u0"], d["u1"], d["u2"], d["u3"]], d["av"])
        b.edge(d["minus"], b"0", d["zero"]); b.edge(d["minus"], b"123456789", d["int"])
        for s in (d["zero"], d["int"], d["frac"], d["exp"]):
            follow(s, c)
        for s in (d["zero"], d["int"]):
            b.edge(s, b".", d["dot"]); b.edge(s, b"eE", d["e"])
        b.edge(d["int"], DIGITS, d["int"])
        b.edge(d["dot"], DIGITS, d["frac"])
        b.edge(d["frac"], DIGITS, d["frac"]); b.edge(d["frac"], b"eE", d["e"])
        b.edge(d["e"], b"+-", d["esign"]); b.edge(d["e"], DIGITS, d["exp"])
        b.edge(d["esign"], DIGITS, d["exp"])
        b.edge(d["exp"], DIGITS, d["exp"])
        for word, names in ((b"true", ("t1", "t2", "t3")), (b"false", ("f1", "f2", "f3", "f4")),
                            (b"null", ("n1", "n2", "n3"))):
            chain = [d[n] for n in names] + [d["av"]]
            for i in range(len(names)):
                b.edge(chain[i], word[i + 1:i + 2], chain[i + 1])
        b.edge(d["av"], WS_JSON, d["av"])
        follow(d["av"], c)

    n_trie = n_states - n_fixed
    n_keys = 20
    keys = _distinct_first_keys(rng, n_keys, n_trie, 4, 24)

    def key_node_common(s):
        # every key-trie node behaves like the generic key string state
        b.edge(s, content, KSTR)
        b.edge(s, b'"', KEND)
        b.edge(s, b"\\", KESC)
    # trie edges are written after the generic ones so they take precedence
    _add_trie(b, KROOT, keys, on_full=lambda s: None, on_other=key_node_common)
    a = b.build(START, max_depth, "json300")
    assert a.n_states == n_states, a.n_states
    return a, keys


# --------------------------------------------------------------------------
# tiny grammars used to pin the oracle (brute force) and as small parity cases
# --------------------------------------------------------------------------
def fig3_expr_pda(max_depth: int = 32) -> Automaton:
    """Fig. 3 (a): E = E | E+E | (E) | int, int = [1-9][0-9]* | 0+, with a ws
    terminal (spaces) allowed between terminals; '(' pushes, ')' pops."""
    b = _Builder()
    OPER = b.state("expect_operand")
    INT = b.state("int_nonzero", accepting=True)
    ZERO = b.state("int_zero", accepting=True)
    AFTER = b.state("after_operand", accepting=True)
    b.edge(OPER, b" ", OPER); b.push(OPER, b"(", 0, OPER)
    b.edge(OPER, b"123456789", INT); b.edge(OPER, b"0", ZERO)
    b.edge(INT, DIGITS, INT)
    b.edge(ZERO, b"0", ZERO)
    for s in (INT, ZERO, AFTER):
        b.edge(s, b" ", AFTER); b.edge(s, b"+", OPER)
        b.pop(s, b")", 0, (AFTER, AFTER, AFTER))
    return b.build(OPER, max_depth, "fig3_expr")


FIG3_VOCAB = [b"0", b"1", b"2", b"12", b")", b"(", b"+", b"+1", b"1 (", b"1 +", b""]


def fig3_vocab() -> Vocab:
    """Fig. 3 (c) vocabulary; the figure spells one token both `1 (` (panels c,
    d) and `1 +` (panel e), so both are present.  The last id is EOS."""
    return Vocab.from_tokens(FIG3_VOCAB, eos_id=len(FIG3_VOCAB) - 1)


def int_regex_dfa() -> Automaton:
    """-?(0|[1-9][0-9]*): 4 live states plus the dead state."""
    b = _Builder()
    START = b.state("start")
    MINUS = b.state("minus")
    ZERO = b.state("zero", accepting=True)
    INT = b.state("int", accepting=True)
    b.edge(START, b"-", MINUS); b.edge(START, b"0", ZERO); b.edge(START, b"123456789", INT)
    b.edge(MINUS, b"0", ZERO); b.edge(MINUS, b"123456789", INT)
    b.edge(INT, DIGITS, INT)
    return b.build(START, 0, "int_regex")


def dyck_ctx_pda(max_depth: int = 3) -> Automaton:
    """Two bracket kinds with context letters: 'c' at top level, 'a' inside
    {...}, 'b' inside [...]; depth <= max_depth; accepting at depth 0.  After a
    closing bracket the state depends on the container that is revealed."""
    b = _Builder()
    TOP = b.state("top", accepting=True)
    OBJ = b.state("in_obj")
    ARR = b.state("in_arr")
    ret = (TOP, OBJ, ARR)
    b.edge(TOP, b"c", TOP); b.edge(OBJ, b"a", OBJ); b.edge(ARR, b"b", ARR)
    for s in (TOP, OBJ, ARR):
        b.push(s, b"{", 0, OBJ)
        b.push(s, b"[", 1, ARR)
    b.pop(OBJ, b"}", 0, ret)
    b.pop(ARR, b"]", 1, ret)
    return b.build(TOP, max_depth, "dyck_ctx")


def dyck2_pda(max_depth: int = 3) -> Automaton:
    """Plain two-bracket Dyck language with letter 'a' anywhere: one scanner
    state, so only the stack top decides whether '}' or ']' may close."""
    b = _Builder()
    TOP = b.state("top", accepting=True)
    b.edge(TOP, b"a", TOP)
    b.push(TOP, b"{", 0, TOP)
    b.push(TOP, b"[", 1, TOP)
    b.pop(TOP, b"}", 0, (TOP, TOP, TOP))
    b.pop(TOP, b"]", 1, (TOP, TOP, TOP))
    return b.build(TOP, max_depth, "dyck2")


def all_strings_vocab(alphabet: bytes, max_len: int, eos: bool = True) -> Vocab:
    """Every string of length 1..max_len over `alphabet` (plus EOS)."""
    import itertools
    toks = []
    for L in range(1, max_len + 1):
        for tup in itertools.product(alphabet, repeat=L):
            toks.append(bytes(tup))
    if eos:
        toks.append(b"")
    return Vocab.from_tokens(toks, eos_id=len(toks) - 1 if eos else -1)


# --------------------------------------------------------------------------
# the five workloads
# --------------------------------------------------------------------------
def workload(config: int) -> Workload:
    root = np.random.SeedSequence(1000 + config)
    r_auto, r_vocab = [np.random.default_rng(s) for s in root.spawn(2)]
    if config == 1:
        a = kv16_dfa()
        uniform = lambda rng, m: rng.integers(1, 9, size=m).astype(np.int64)
        alpha = np.frombuffer(CFG1_ALPHABET, dtype=np.uint8)
        v = random_vocab(r_vocab, 1024, CFG1_ALPHABET, uniform, lambda rng, n: alpha[rng.integers(0, alpha.size, n)])
        return Workload(1, "kv16_v1024_b1", a, v, batch=1, steps=64, logits_dtype="f32", logits_sigma=1.0,
                        want_logprobs=False,
                        description="16-state key/value DFA, V=1024, batch 1, fp32 logits N(0,1)")
    if config == 2:
        a, _ = kv200_dfa(r_auto)
        v = random_vocab(r_vocab, 32000, bytes(range(256)), geometric_lengths(4.0, 16), _mixed_bytes)
        return Workload(2, "kv200_v32000_b32", a, v, batch=32, steps=256, logits_dtype="bf16", logits_sigma=2.0,
                        want_logprobs=False,
                        description="200-state 8-key JSON-like DFA, V=32000, batch 32, bf16 logits N(0,2)")
    if config in (3, 4):
        Q = 5000 if config == 3 else 20000
        a = random_sparse_dfa(r_auto, Q)
        v = random_vocab(r_vocab, 128256, bytes(range(256)), geometric_lengths(4.5, 32), _mixed_bytes)
        if config == 3:
            return Workload(3, "sparse5000_v128256_b256", a, v, batch=256, steps=64, logits_dtype="bf16",
                            logits_sigma=3.0, want_logprobs=False,
                            description="random sparse DFA Q=5000, V=128256, batch 256, bf16 logits N(0,3)")
        return Workload(4, "precompute_sparse20000_v128256", a, v, batch=Q, steps=1, logits_dtype="bf16",
                        logits_sigma=3.0, want_logprobs=False,
                        description="state x token table: random sparse DFA Q=20000 x V=128256")
    if config == 5:
        a, _ = json_pda(r_auto)
        v = random_vocab(r_vocab, 152064, bytes(range(256)), geometric_lengths(4.0, 32), _mixed_bytes)
        return Workload(5, "json300_pda_v152064_b128", a, v, batch=128, steps=64, logits_dtype="bf16",
                        logits_sigma=3.0, want_logprobs=True,
                        description="300-state JSON lexer + bracket stack (depth<=32), V=152064, batch 128, "
                                    "bf16 logits N(0,3), log-probs")
    raise ValueError(f"unknown config {config}")
