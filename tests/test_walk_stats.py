"""The oracle's count of the work of the plain mask definition (bytes walked per
check), which states the algorithmic units of the mask-walk roofline.  Pinned by
closed forms and hand-walked tokens; the stored per-workload figures are checked
against a fresh oracle run."""
import json
import os

import numpy as np

from paper_2403_06988_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "walk_stats.json")


def _two_state(target_of_live_state: int) -> synth.Automaton:
    """States 0 (dead) and 1; every byte from 1 goes to `target_of_live_state`."""
    delta = np.zeros((2, 256), np.int32)
    delta[1, :] = target_of_live_state
    live = np.array([0, 1], np.uint8)
    return synth.Automaton(delta=delta, live=live, accepting=live.copy(), start=1, rules=None, max_depth=0)


def test_every_byte_walked_when_nothing_dies(oracle_lib):
    toks = [b"a", b"bc", b"", b"defg", b"\xff" * 9]
    vocab = synth.Vocab.from_tokens(toks + [b""], eos_id=len(toks))
    P = oracle_lib.Problem.from_parts(_two_state(1), vocab)
    states = np.ones(3, np.int32)
    assert P.walk_steps(states) == 3 * (1 + 2 + 4 + 9)     # empty and EOS tokens take no step


def test_one_step_per_token_when_the_first_byte_dies(oracle_lib):
    toks = [b"a", b"bc", b"", b"defg"]
    P = oracle_lib.Problem.from_parts(_two_state(0), synth.Vocab.from_tokens(toks))
    assert P.walk_steps(np.ones(5, np.int32)) == 5 * 3
    assert P.walk_steps(np.zeros(5, np.int32)) == 5 * 3      # the dead state rejects at the first byte too
    assert P.walk_steps(np.full(5, 7, np.int32)) == 0         # out-of-range rows are invalid: no walk


def test_hand_walked_tokens_on_the_integer_regex(oracle_lib):
    a = synth.int_regex_dfa()                                 # -?(0|[1-9][0-9]*)
    cases = {b"-0": 2, b"00": 2, b"a0": 1, b"-12": 3, b"1-": 2, b"--": 2, b"7": 1}
    vocab = synth.Vocab.from_tokens(list(cases))
    P = oracle_lib.Problem.from_parts(a, vocab)
    assert P.walk_steps(np.array([a.start], np.int32)) == sum(cases.values())


def test_stored_figures_match_the_oracle(oracle_lib):
    with open(GOLDEN) as f:
        stored = json.load(f)
    w = synth.workload(1)
    P = oracle_lib.Problem.from_workload(w)
    states, _ = w.initial_configs(part=2)
    fresh = P.walk_steps(states) / (w.batch * w.vocab.n_tokens)
    assert stored[w.name]["walk_steps_per_check_step0"] == fresh
    for rec in stored.values():
        assert rec["walk_steps_per_check_mean"] >= 1.0 or rec["config"] == 1
