"""Checks of the seeded workload generators against independent descriptions.

* live == co-reachable to acceptance, recomputed by reverse BFS;
* the config-1 DFA equals a regex of its language;
* the config-5 JSON lexer + bracket stack accepts json.dumps output and
  everything it accepts parses with Python's json module as an object;
* every configuration reached by an allowed token can still complete
  (operational rule == prefix viability, Sec. 3.5 at k = infinity).
"""
import json
import re
from collections import deque

import numpy as np
import pytest

from paper_2403_06988_gb300 import synth


def coreachable(a: synth.Automaton) -> np.ndarray:
    Q = a.n_states
    succ_extra = {}
    if a.rules is not None:
        for r in a.rules:
            if r["kind"] == synth.RULE_POP:
                succ_extra.setdefault(int(r["state"]), set()).update(
                    {int(r["next_if_empty"]), int(r["next_if_top0"]), int(r["next_if_top1"])})
    good = a.accepting.astype(bool).copy()
    while True:
        hit = good[a.delta].any(axis=1)
        for s, ts in succ_extra.items():
            hit[s] |= any(good[t] for t in ts if t != 0)
        hit[0] = False
        new = good | hit
        if (new == good).all():
            return good
        good = new


@pytest.mark.parametrize("config", [1, 2, 3, 5])
def test_live_is_coreachable(config):
    a = synth.workload(config).automaton
    assert (coreachable(a) == a.live.astype(bool)).all()
    assert a.live[0] == 0 and (a.delta[0] == 0).all()
    assert not (a.accepting.astype(bool) & ~a.live.astype(bool)).any()


def test_sparse_dfa_shape():
    a = synth.workload(3).automaton
    live_bytes = (a.delta[1:] != 0).sum(axis=1)
    assert (live_bytes == 64).all()                       # 8 live classes x 8 bytes
    assert a.accepting.sum() == 500


def test_vocab_shapes():
    for config, V, maxlen in ((1, 1024, 8), (2, 32000, 16), (3, 128256, 32), (5, 152064, 32)):
        w = synth.workload(config)
        toks = w.vocab.tokens()
        assert len(toks) == V and w.vocab.eos_id == V - 1 and toks[-1] == b""
        assert len(set(toks)) == V
        assert max(len(t) for t in toks) <= maxlen
        if config >= 2:
            assert toks[:256] == [bytes([c]) for c in range(256)]


CFG1_VAL = r'(?:0|[1-9][0-9]*|[a-z][a-z0-9]*|"[a-z0-9 ]*")'
CFG1_PAIR = r'"[a-z][a-z0-9]*" *: *' + CFG1_VAL + r' *'
CFG1_RE = re.compile((r' *\{ *(?:' + CFG1_PAIR + r'(?:, *' + CFG1_PAIR + r')*)?\} *').encode())


def dfa_accepts(a, s: bytes) -> bool:
    q = a.start
    for c in s:
        q = a.delta[q, c]
        if q == 0:
            return False
    return bool(a.accepting[q])


def test_config1_dfa_matches_regex():
    a = synth.workload(1).automaton
    rng = np.random.default_rng(0)
    alpha = b'{}": ,a1z0'
    n_acc = 0
    for _ in range(20000):
        L = int(rng.integers(1, 18))
        s = bytes(alpha[i] for i in rng.integers(0, len(alpha), L))
        assert dfa_accepts(a, s) == bool(CFG1_RE.fullmatch(s)), s
    for _ in range(3000):        # random members built from the regex's pieces
        pairs = []
        for _ in range(int(rng.integers(0, 4))):
            key = "k" + "".join(rng.choice(list("ab09"), int(rng.integers(0, 3))))
            val = rng.choice(["0", "42", "x1", '""', '"a b"'])
            pairs.append(f'"{key}"' + " " * int(rng.integers(0, 2)) + ":" + " " * int(rng.integers(0, 2)) + val)
        s = (" {" + ", ".join(pairs) + "} ").encode()
        assert dfa_accepts(a, s), s
        n_acc += 1
    assert n_acc == 3000


# --------------------------------------------------------------------------
# config 5: JSON lexer + bracket stack
# --------------------------------------------------------------------------
class PdaRunner:
    """Test-side byte stepper (independent of the oracle) for acceptance checks."""

    def __init__(self, a):
        self.a = a
        self.rule = {(int(r["state"]), int(r["byte"])): r for r in a.rules}

    def step(self, s, stk, c):
        r = self.rule.get((s, c))
        if r is None:
            t = int(self.a.delta[s, c])
            return (t, stk) if t and self.a.live[t] else None
        if r["kind"] == synth.RULE_PUSH:
            if len(stk) == self.a.max_depth:
                return None
            t = int(self.a.delta[s, c])
            return (t, stk + (int(r["sym"]),)) if t else None
        if not stk or stk[-1] != r["sym"]:
            return None
        stk = stk[:-1]
        t = int(r["next_if_empty"] if not stk else (r["next_if_top0"] if stk[-1] == 0 else r["next_if_top1"]))
        return (t, stk) if t and self.a.live[t] else None

    def accepts(self, data: bytes) -> bool:
        s, stk = self.a.start, ()
        for c in data:
            nxt = self.step(s, stk, c)
            if nxt is None:
                return False
            s, stk = nxt
        return bool(self.a.accepting[s]) and not stk

    def outcomes(self, s):
        """Distinct moves out of state s: one representative byte per outcome."""
        if not hasattr(self, "_out"):
            self._out = {}
        if s not in self._out:
            seen, reps = set(), []
            for c in range(256):
                r = self.rule.get((s, c))
                if r is None:
                    key = ("step", int(self.a.delta[s, c]))
                elif r["kind"] == synth.RULE_PUSH:
                    key = ("push", int(r["sym"]), int(self.a.delta[s, c]))
                else:
                    key = ("pop", int(r["sym"]), int(r["next_if_empty"]), int(r["next_if_top0"]),
                           int(r["next_if_top1"]))
                if key not in seen:
                    seen.add(key)
                    reps.append(c)
            self._out[s] = reps
        return self._out[s]

    def completable(self, s, stk) -> bool:
        """BFS to (accepting, empty) that may push at most one level above the start depth."""
        limit = min(self.a.max_depth, len(stk) + 1)
        seen = {(s, stk)}
        dq = deque([(s, stk)])
        while dq:
            s, stk = dq.popleft()
            if self.a.accepting[s] and not stk:
                return True
            for c in self.outcomes(s):
                nxt = self.step(s, stk, c)
                if nxt is not None and len(nxt[1]) <= limit and nxt not in seen:
                    seen.add(nxt)
                    dq.append(nxt)
        return False


def random_json(rng, depth=0):
    k = int(rng.integers(0, 7 if depth < 4 else 4))
    if k == 0:
        return {}
    if k == 1 and depth < 6:
        return {f"k{int(rng.integers(0, 9))}": random_json(rng, depth + 1) for _ in range(int(rng.integers(1, 4)))}
    if k == 2 and depth < 6:
        return [random_json(rng, depth + 1) for _ in range(int(rng.integers(0, 4)))]
    if k == 3:
        return "".join(rng.choice(list('ab "\\/é\n x'), int(rng.integers(0, 6))))
    if k == 4:
        return int(rng.integers(-1000, 1000))
    if k == 5:
        return float(rng.standard_normal() * 10 ** int(rng.integers(-8, 8)))
    return [True, False, None][int(rng.integers(0, 3))]


def test_config5_accepts_python_json():
    a = synth.workload(5).automaton
    run = PdaRunner(a)
    rng = np.random.default_rng(1)
    for i in range(400):
        obj = {"root": random_json(rng)} if i % 2 else {f"k{j}": random_json(rng) for j in range(3)}
        for kw in ({}, {"indent": 1}, {"separators": (",", ":")}, {"ensure_ascii": False}):
            text = json.dumps(obj, **kw).encode()
            assert run.accepts(text), text


def test_config5_accepted_strings_are_json_objects():
    a = synth.workload(5).automaton
    run = PdaRunner(a)
    rng = np.random.default_rng(2)
    n_ok = 0
    for _ in range(300):
        s, stk, out = a.start, (), bytearray()
        for _ in range(120):
            if a.accepting[s] and not stk and rng.random() < 0.3:
                break
            opts = [(c, run.step(s, stk, c)) for c in range(256)]
            opts = [(c, n) for c, n in opts if n is not None]
            if len(stk) > 3:      # steer towards closing
                closing = [(c, n) for c, n in opts if len(n[1]) < len(stk)]
                opts = closing or opts
            c, (s, stk) = opts[int(rng.integers(0, len(opts)))]
            out.append(c)
        if a.accepting[s] and not stk:
            val = json.loads(out.decode("latin-1"), strict=False)
            assert isinstance(val, dict)
            n_ok += 1
    assert n_ok > 30


def test_config5_reachable_configurations_complete(oracle_lib):
    w = synth.workload(5)
    a = w.automaton
    run = PdaRunner(a)
    P = oracle_lib.Problem.from_workload(w)
    states, stacks = w.initial_configs(batch=12)
    rng = np.random.default_rng(4)
    checked = 0
    for s, st in zip(states, stacks):
        assert run.completable(int(s), tuple(synth.unpack_stack(int(st))))
        for t in rng.integers(0, w.vocab.n_tokens - 1, size=40):
            r, s2, w2 = P.check(int(s), int(st), int(t))
            if r == 1:
                assert run.completable(s2, tuple(synth.unpack_stack(w2)))
                checked += 1
    assert checked > 20
