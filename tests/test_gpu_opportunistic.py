"""Opportunistic masking (Sec. 3.5, further optimisations): the unmasked argmax
is proposed and checked with one walk; only rejected rows get a mask.  The
tokens must equal the masked greedy decode of the oracle, bit for bit.
Output buffers start as 0xAB bytes (tests/poison.py)."""
import functools
import os

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

from paper_2403_06988_gb300 import Domino, synth  # noqa: E402
from paper_2403_06988_gb300 import _binding as B  # noqa: E402
from poison import assert_exact  # noqa: E402

NT = os.cpu_count() or 1


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2403_06988_gb300 import build
    build.build()


@functools.lru_cache(maxsize=None)
def workload(config):
    return synth.workload(config)


@functools.lru_cache(maxsize=None)
def handle(config):
    w = workload(config)
    return Domino.from_parts(w.automaton, w.vocab, device=0)


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def logits_tensor(x):
    return dev(x.view(np.int16)).view(torch.bfloat16) if x.dtype == np.uint16 else dev(x)


def oracle_greedy(config, states, stacks, lg):
    import oracle
    w = workload(config)
    P = oracle.Problem.from_workload(w)
    sk = stacks if w.automaton.rules is not None else None
    m, _, _ = P.step_mask(states, sk, n_threads=NT)
    arg, _, _ = oracle.mask_logits(lg, m)
    V = w.vocab.n_tokens
    ones = np.full_like(m, 0xFFFFFFFF)
    if V % 32:
        ones[:, -1] = (1 << (V % 32)) - 1
    prop, _, _ = oracle.mask_logits(lg, ones)
    accepted = (m[np.arange(len(prop)), prop // 32] >> (prop % 32)) & 1
    return arg, m, int((accepted == 0).sum())


def biased(lg, m, V, bias):
    """Logits of an obedient model: +bias on every allowed token (float32 or bf16 bits)."""
    bits = np.unpackbits(m.view(np.uint8), axis=1, bitorder="little")[:, :V].astype(bool)
    x = synth.bf16_bits_to_f32(lg) if lg.dtype == np.uint16 else lg.copy()
    x = x + bias * bits
    return synth.f32_to_bf16_bits(x) if lg.dtype == np.uint16 else x.astype(np.float32)


@pytest.mark.parametrize("config", [1, 2, 3, 5])
@pytest.mark.parametrize("obedient", [False, True])
def test_opportunistic_matches_masked_greedy(config, obedient):
    w = workload(config)
    states, stacks = w.initial_configs()
    lg = w.logits(1)
    if obedient:
        _, m, _ = oracle_greedy(config, states, stacks, lg)
        lg = biased(lg, m, w.vocab.n_tokens, 20.0)
    want, _, n_rej = oracle_greedy(config, states, stacks, lg)
    d = handle(config)
    sk = dev(stacks.view(np.int64)) if w.automaton.rules is not None else None
    tok, n_fb = d.opportunistic_step(logits_tensor(lg), dev(states), sk)
    assert_exact(tok, np.asarray(want, np.int32), "tokens")
    assert int(n_fb.item()) == n_rej
    if obedient:
        assert n_rej == int((want < 0).sum())      # only rows with nothing allowed fall back
    assert d.device_error() == 0


def test_opportunistic_decode_loop_with_advance():
    import oracle
    config, steps = 2, 24
    w = workload(config)
    P = oracle.Problem.from_workload(w)
    d = handle(config)
    states, _ = w.initial_configs()
    st = dev(states)
    s_o = states.copy()
    for i in range(steps):
        lg = w.logits(50 + i)
        m_o, _, _ = P.step_mask(s_o, None, n_threads=NT)
        if i % 2:
            lg = biased(lg, m_o, w.vocab.n_tokens, 6.0)   # alternate: mostly rejected / mostly accepted
        tok, _ = d.opportunistic_step(logits_tensor(lg), st)
        d.advance(st, None, tok)
        a_o, _, _ = oracle.mask_logits(lg, m_o)
        s_o, _, _ = P.advance(s_o, None, a_o, w.automaton.start)
        assert_exact(tok, np.asarray(a_o, np.int32), f"tokens, step {i}")
        assert (st.cpu().numpy() == s_o).all(), i


def test_opportunistic_invalid_rows():
    w = workload(2)
    d = handle(2)
    Q = w.automaton.n_states
    st = dev(np.array([-5, Q, 0, 1], np.int32))
    tok, n_fb = d.opportunistic_step(logits_tensor(w.logits(0, batch=4)), st)
    t = tok.cpu().numpy()
    assert (t[:3] == -1).all()
    assert int(n_fb.item()) >= 3
    assert d.device_error() == B.DEVERR_BAD_STATE


def test_opportunistic_more_rows_than_one_logits_pass():
    """4100 rows: the fallback list spans two passes of the logits kernel."""
    import oracle
    w = workload(1)
    P = oracle.Problem.from_workload(w)
    d = handle(1)
    rng = np.random.default_rng(11)
    states = rng.choice(np.nonzero(w.automaton.live)[0], size=4100).astype(np.int32)
    x = (rng.standard_normal((4100, w.vocab.n_tokens)) * 2).astype(np.float32)
    m, _, _ = P.step_mask(states, None, n_threads=NT)
    allowed_rows = np.unpackbits(m.view(np.uint8), axis=1, bitorder="little")[:, :w.vocab.n_tokens].sum(axis=0)
    x[:, int(np.argmin(allowed_rows))] += 50.0          # a token almost never allowed wins every proposal
    want, _, _ = oracle.mask_logits(x, m)
    tok, n_fb = d.opportunistic_step(dev(x), dev(states))
    assert_exact(tok, np.asarray(want, np.int32), "tokens")
    assert int(n_fb.item()) > 4096

