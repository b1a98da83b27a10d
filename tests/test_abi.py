"""The C ABI without a GPU: library loads, every declared entry point is
exported, host-only handles validate and preprocess loads, and compute calls
fail loudly instead of falling back to the CPU."""
import ctypes

import numpy as np
import pytest

from paper_2403_06988_gb300 import _binding as B
from paper_2403_06988_gb300 import build as build_mod
from paper_2403_06988_gb300 import synth


@pytest.fixture(scope="module")
def lib():
    build_mod.build()
    return B.lib()


def test_every_declared_symbol_is_exported(lib):
    names = B.header_symbols()
    assert len(names) >= 13
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) >= set(B._SIGS) | {"domino_status_string"}


def test_status_strings(lib):
    assert B.status_string(0) == "ok"
    for code in range(-1, -7, -1):
        assert B.status_string(code) != "unknown status"
    assert B.status_string(-99) == "unknown status"


def host_handle(config=None, automaton=None, vocab=None):
    h = B.domino_create(-1)
    if config is not None:
        w = synth.workload(config)
        automaton, vocab = w.automaton, w.vocab
    if vocab is not None:
        B.domino_load_vocab(h, vocab.data, vocab.offsets, vocab.n_tokens, vocab.eos_id)
    if automaton is not None:
        a = automaton
        B.domino_load_automaton(h, a.delta, a.n_states, a.live, a.accepting, a.start, a.rules, None, a.max_depth)
    return h


def columns(a: synth.Automaton):
    """Per byte: the tuple of (target, rule) over all states."""
    rule = {}
    if a.rules is not None:
        for r in a.rules:
            rule[(int(r["state"]), int(r["byte"]))] = tuple(int(x) for x in r)[2:]
    cols = []
    for c in range(256):
        cols.append(tuple((int(a.delta[q, c]) if a.live[a.delta[q, c]] else 0, rule.get((q, c)))
                          for q in range(a.n_states)))
    return cols


@pytest.mark.parametrize("config", [1, 2, 3, 5])
def test_byte_classes_partition(lib, config):
    w = synth.workload(config)
    h = host_handle(config)
    try:
        info = B.domino_get_info(h)
        cls = B.domino_get_byte_classes(h)
        cols = columns(w.automaton)
        assert info["n_classes"] == len(set(cols)) == int(cls.max()) + 1
        for c1 in range(256):
            for c2 in range(c1 + 1, 256):
                assert (cls[c1] == cls[c2]) == (cols[c1] == cols[c2])
        assert info["n_tokens"] == w.vocab.n_tokens and info["n_states"] == w.automaton.n_states
        assert info["has_stack"] == (1 if w.automaton.rules is not None else 0)
        if config == 3:
            assert info["n_classes"] == 32
    finally:
        B.domino_destroy(h)


def test_compute_on_host_handle_refuses(lib):
    h = host_handle(1)
    try:
        with pytest.raises(B.DominoError) as e:
            B.domino_step_mask(h, 0, None, 1, 0, None, stream=0)
        assert e.value.status == -6
        with pytest.raises(B.DominoError) as e:
            B.domino_mask_logits(h, 0, 0, 1, 1024, 0, 0, stream=0)
        assert e.value.status == -6
        with pytest.raises(B.DominoError) as e:
            B.domino_get_device_error(h, stream=0)
        assert e.value.status == -6
    finally:
        B.domino_destroy(h)


def _bad_load(a, **kw):
    h = B.domino_create(-1)
    try:
        args = dict(delta=a.delta, n_states=a.n_states, live=a.live, accepting=a.accepting, start_state=a.start,
                    rules=a.rules, n_rules=None, max_depth=a.max_depth)
        args.update(kw)
        with pytest.raises(B.DominoError) as e:
            B.domino_load_automaton(h, **args)
        return e.value.status
    finally:
        B.domino_destroy(h)


def test_automaton_validation(lib):
    a = synth.fig3_expr_pda()
    d = a.delta.copy(); d[0, 5] = 1
    assert _bad_load(a, delta=d) == -1                       # state 0 not absorbing
    lv = a.live.copy(); lv[0] = 1
    assert _bad_load(a, live=lv) == -1                       # state 0 live
    d = a.delta.copy(); d[2, 7] = 9
    assert _bad_load(a, delta=d) == -1                       # id out of range
    acc = a.accepting.copy(); lv = a.live.copy(); lv[2] = 0
    assert _bad_load(a, live=lv) == -1                       # accepting but not live / live reached from dead
    assert _bad_load(a, max_depth=33) == -1
    assert _bad_load(a, start_state=5) == -1
    r = a.rules.copy(); r[0]["sym"] = 2
    assert _bad_load(a, rules=r) == -1
    r = np.concatenate([a.rules, a.rules[:1]])
    assert _bad_load(a, rules=r) == -1                       # two rules on one (state, byte)
    r = a.rules.copy(); r[0]["state"] = 0
    assert _bad_load(a, rules=r) == -1                       # a rule on the dead state
    r = a.rules.copy(); r[0]["kind"] = 3
    assert _bad_load(a, rules=r) == -1
    # a non-live state whose successor is live
    d = np.zeros((3, 256), np.int32); d[1, ord("a")] = 2; d[2, ord("a")] = 1
    lv = np.array([0, 0, 1], np.uint8)
    assert _bad_load(a, delta=d, n_states=3, live=lv, accepting=np.array([0, 0, 1], np.uint8), start_state=2,
                     rules=None, max_depth=0) == -1


def test_vocab_validation(lib):
    h = B.domino_create(-1)
    try:
        data = np.frombuffer(b"abcd", np.uint8)
        for offs, eos in (([0, 2, 1, 4], -1), ([1, 2, 3, 4], -1), ([0, 1, 2, 4], 3), ([0, 1, 2, 4], -2)):
            with pytest.raises(B.DominoError):
                B.domino_load_vocab(h, data, np.array(offs, np.int64), 3, eos)
        B.domino_load_vocab(h, data, np.array([0, 1, 2, 4], np.int64), 3, -1)
        assert B.domino_get_info(h)["max_token_len"] == 2
    finally:
        B.domino_destroy(h)


def test_stack_rule_layout():
    assert ctypes.sizeof(B.StackRule) == 20 == synth.RULE_DTYPE.itemsize
