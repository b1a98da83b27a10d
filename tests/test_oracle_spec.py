"""Pins of the oracle's count-based speculation (Sec. 3.6).

The count model P(t | alpha, beta) = #chose(t) / #reached is checked on hand
examples whose proposals follow from the counts by inspection; the
structural rules (a proposal is always allowed from its chain configuration,
the chain follows the walk, the update is order independent, the parser
sub-state beta separates stack tops) on random runs."""
import numpy as np
import pytest

import oracle
from paper_2403_06988_gb300 import synth


def tok_vocab(tokens, eos=True):
    return synth.Vocab.from_tokens(list(tokens) + ([b""] if eos else []), eos_id=len(tokens) if eos else -1)


def test_most_frequent_choice_above_the_threshold():
    a = synth.int_regex_dfa()                       # -?(0|[1-9][0-9]*)
    v = tok_vocab([b"1", b"2", b"12", b"-", b"0"])
    P = oracle.Problem.from_parts(a, v)
    sp = oracle.Spec(P)
    start = np.array([a.start], np.int32)
    for t in [0, 0, 0, 1]:                          # "1" three times, "2" once from the start state
        sp.update(start, None, np.array([t], np.int32))
    prop, n, cs, _ = sp.propose(start, None, 4, 500)
    assert n[0] == 1 and prop[0, 0] == 0 and (prop[0, 1:] == -1).all()   # 3/4 >= 0.5; INT never reached
    r, s_int, _ = P.check(a.start, 0, 0)
    assert cs[0, 0] == a.start and (cs[0, 1:] == s_int).all()
    prop, n, _, _ = sp.propose(start, None, 4, 800)                      # 3/4 < 0.8
    assert n[0] == 0 and (prop == -1).all()
    prop, n, _, _ = sp.propose(start, None, 4, 750)                      # 3/4 >= 0.75 exactly
    assert n[0] == 1


def test_chains_continue_through_reached_states_and_ties_take_the_lowest_id():
    a = synth.int_regex_dfa()
    v = tok_vocab([b"1", b"2", b"12", b"3"])
    P = oracle.Problem.from_parts(a, v)
    sp = oracle.Spec(P)
    _, s_int, _ = P.check(a.start, 0, 0)
    st = np.array([a.start], np.int32)
    si = np.array([s_int], np.int32)
    sp.update(st, None, np.array([2], np.int32))   # from start: "12" once, "3" once -> tie: lowest id "12"
    sp.update(st, None, np.array([3], np.int32))
    for _ in range(2):
        sp.update(si, None, np.array([1], np.int32))   # from INT: "2" twice
    prop, n, cs, _ = sp.propose(st, None, 3, 500)
    assert list(prop[0]) == [2, 1, 1] and n[0] == 3
    assert (cs[0] == s_int).sum() == 3 and cs[0, 0] == a.start


def test_eos_is_proposed_only_where_allowed_and_ends_the_chain():
    a = synth.int_regex_dfa()
    v = tok_vocab([b"1"])
    eos = v.eos_id
    P = oracle.Problem.from_parts(a, v)
    sp = oracle.Spec(P)
    _, s_int, _ = P.check(a.start, 0, 0)
    si = np.array([s_int], np.int32)
    sp.update(si, None, np.array([eos], np.int32))
    prop, n, cs, _ = sp.propose(si, None, 3, 100)
    assert n[0] == 1 and prop[0, 0] == eos and (cs[0] == s_int).all()
    st = np.array([a.start], np.int32)                # EOS counted at start, where it is not allowed
    sp.update(st, None, np.array([eos], np.int32))
    prop, n, _, _ = sp.propose(st, None, 3, 100)
    assert n[0] == 0


def test_stack_top_is_part_of_the_key():
    a = synth.dyck2_pda(3)
    v = tok_vocab([b"{", b"[", b"}", b"]", b"a"])
    P = oracle.Problem.from_parts(a, v)
    sp = oracle.Spec(P)
    _, s1, w_obj = P.check(a.start, 0, 0)          # after "{": top 0
    _, s2, w_arr = P.check(a.start, 0, 1)          # after "[": top 1
    assert s1 == s2 and w_obj != w_arr             # one scanner state, two parser sub-states
    sp.update(np.array([s1], np.int32), np.array([w_obj], np.uint64), np.array([2], np.int32))   # "}"
    sp.update(np.array([s2], np.int32), np.array([w_arr], np.uint64), np.array([3], np.int32))   # "]"
    prop, n, _, ck = sp.propose(np.array([s1, s2], np.int32), np.array([w_obj, w_arr], np.uint64), 2, 500)
    assert prop[0, 0] == 2 and prop[1, 0] == 3
    assert ck[0, 1] == 0 and ck[1, 1] == 0         # both closed back to the empty stack


@pytest.mark.parametrize("config", [2, 5])
def test_random_runs_structural_rules(config):
    w = synth.workload(config)
    P = oracle.Problem.from_workload(w)
    has_stack = w.automaton.rules is not None
    rng = np.random.default_rng(config)
    states, stacks = w.initial_configs(batch=24)
    sk = stacks if has_stack else None
    sp1, sp2 = oracle.Spec(P), oracle.Spec(P)
    for step in range(6):
        m, _, _ = P.step_mask(states, sk, n_threads=4)
        arg, _, _ = oracle.mask_logits(w.logits(step, batch=24), m)
        order = rng.permutation(len(states))
        sp1.update(states, sk, arg)
        sp2.update(states[order], None if sk is None else sk[order], arg[order])
        states, sk2, _ = P.advance(states, sk, arg, w.automaton.start)
        sk = sk2 if has_stack else None
    s = 5
    r1 = sp1.propose(states, sk, s, 0)
    r2 = sp2.propose(states, sk, s, 0)
    for x, y in zip(r1, r2):
        assert (x is None and y is None) or (x == y).all()   # order of updates does not matter
    prop, n, cs, ck = r1
    assert n.max() > 0
    for b in range(len(states)):
        for i in range(n[b]):
            t = int(prop[b, i])
            r, ns, nw = P.check(int(cs[b, i]), int(ck[b, i]) if ck is not None else 0, t)
            assert r == 1                          # every proposal is allowed where it is made
            if t != w.vocab.eos_id:
                assert ns == cs[b, i + 1] and (ck is None or nw == ck[b, i + 1])


def test_accept_counts_the_agreeing_prefix():
    prop = np.array([[4, 5, 6], [4, 5, 6], [7, -1, -1]], np.int32)
    n = np.array([3, 3, 1], np.int32)
    dec = np.array([[4, 5, 9, 1], [4, 5, 6, 2], [7, 3, 3, 3]], np.int32)
    assert list(oracle.spec_accept(prop, n, dec)) == [2, 3, 1]
