"""domino_step_decode: the mask step with the masked greedy decode folded into
it, against the oracle (mask and argmax bit-exact, lse within 1e-3), with
device and pinned host logits, a ragged vocabulary and invalid rows.  Output
buffers start as 0xAB bytes (tests/poison.py)."""
import functools
import os

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

from paper_2403_06988_gb300 import Domino, synth  # noqa: E402
from paper_2403_06988_gb300 import _binding as B  # noqa: E402
import poison  # noqa: E402
from poison import assert_exact, assert_no_poison  # noqa: E402

TOL = 1e-3
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


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def run(d, states, stacks, logits, dtype, stride, batch, W, V=None):
    mask = poison.empty((batch, W), torch.int32)
    arg = poison.empty(batch, torch.int32)
    lse = poison.empty(batch, torch.float32)
    lp = poison.empty((batch, V), torch.float32) if V else None
    B.domino_step_decode(d.h, states, stacks, batch, logits, dtype, stride, mask, arg, lse, lp)
    torch.cuda.synchronize()
    out = (mask.cpu().numpy().view(np.uint32), arg.cpu().numpy(), lse.cpu().numpy())
    return out + ((lp.cpu().numpy(),) if V else ())


def check(P, states, stacks, lg, V, m, a, l, lp=None):
    import oracle
    m_o, _, _ = P.step_mask(states, stacks, n_threads=NT)
    a_o, l_o, lp_o = oracle.mask_logits(lg, m_o, n_tokens=V, want_logprobs=lp is not None, n_threads=NT)
    assert_exact(m, m_o, "mask")
    assert_exact(a, np.asarray(a_o, np.int32), "argmax")
    assert_no_poison(l, "lse")
    fin = np.isfinite(l_o)
    assert (np.isfinite(l) == fin).all()
    assert np.abs(l[fin] - l_o[fin]).max(initial=0) < TOL
    if lp is not None:
        assert_no_poison(lp, "log-probs")
        fin = np.isfinite(lp_o)
        assert (np.isfinite(lp) == fin).all()
        assert np.abs(lp[fin] - lp_o[fin]).max(initial=0) < TOL


@pytest.mark.parametrize("config,pinned", [(1, False), (2, False), (3, False), (3, True), (5, False), (5, True)])
def test_step_decode_matches_oracle(config, pinned):
    import oracle
    w = workload(config)
    P = oracle.Problem.from_workload(w)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    states, stacks = w.initial_configs()
    has_stack = w.automaton.rules is not None
    lg = w.logits(7)
    host = torch.from_numpy(lg.view(np.int16) if lg.dtype == np.uint16 else lg)
    t = host.pin_memory() if pinned else host.cuda()
    dt = B.DTYPE_BF16 if lg.dtype == np.uint16 else B.DTYPE_F32
    V = w.vocab.n_tokens
    want_lp = config in (2, 5)
    res = run(d, dev(states), dev(stacks.view(np.int64)) if has_stack else None, t.data_ptr(), dt, V, len(states),
              d.info()["n_words"], V if want_lp else None)
    check(P, states, stacks if has_stack else None, lg, V, *res)
    d.close()


@pytest.mark.parametrize("stride", [1008, 1003])
def test_step_decode_ragged_vocabulary_padded_rows_and_invalid_states(stride):
    """V = 1003 (a partial last mask word); rows padded to 1008 elements (16-byte
    aligned rows: the fused kernel) or packed at 1003 (the two-kernel path)."""
    import oracle
    rng = np.random.default_rng(17)
    a_ = synth.int_regex_dfa()
    alphabet = b"-0123456789x"
    toks, seen = [], set()
    while len(toks) < 1002:
        n = int(rng.integers(1, 7))
        t = bytes(alphabet[i] for i in rng.integers(0, len(alphabet), n))
        if t not in seen:
            seen.add(t)
            toks.append(t)
    vocab = synth.Vocab.from_tokens(toks + [b""], eos_id=1002)
    V, batch = 1003, 40
    P = oracle.Problem.from_parts(a_, vocab)
    d = Domino.from_parts(a_, vocab, device=0)
    live = np.nonzero(a_.live)[0]
    states = rng.choice(live, size=batch).astype(np.int32)
    states[3] = -1
    states[7] = a_.n_states          # invalid rows: empty masks, argmax -1
    x = (rng.standard_normal((batch, stride)) * 2).astype(np.float32)
    bf = synth.f32_to_bf16_bits(x)
    lg_dev = dev(bf.view(np.int16))   # held: the outputs must not reuse its memory
    m, a, l, lp = run(d, dev(states), None, lg_dev.data_ptr(), B.DTYPE_BF16, stride, batch, d.info()["n_words"], V)
    check(P, states, None, bf, V, m, a, l, lp)
    assert a[3] == -1 and a[7] == -1
    assert d.device_error() == B.DEVERR_BAD_STATE
    d.close()


@pytest.mark.parametrize("config", [3, 5])
def test_step_decode_equal_logits_pick_the_lowest_allowed_token(config):
    """Every logit equal: the argmax is each row's first allowed token and
    lse = c + ln(#allowed), across sparse and dense row windows."""
    import oracle
    w = workload(config)
    P = oracle.Problem.from_workload(w)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    states, stacks = w.initial_configs(batch=64)
    has_stack = w.automaton.rules is not None
    V = w.vocab.n_tokens
    bf = np.full((len(states), V), synth.f32_to_bf16_bits(np.array([1.5], np.float32))[0], np.uint16)
    lg_dev = dev(bf.view(np.int16))
    m, a, l = run(d, dev(states), dev(stacks.view(np.int64)) if has_stack else None, lg_dev.data_ptr(),
                  B.DTYPE_BF16, V, len(states), d.info()["n_words"])
    check(P, states, stacks if has_stack else None, bf, V, m, a, l)
    bits = np.unpackbits(m.view(np.uint8), bitorder="little").reshape(len(states), -1)[:, :V]
    for b in range(len(states)):
        allowed = np.nonzero(bits[b])[0]
        if len(allowed):
            assert a[b] == allowed[0]
            assert abs(l[b] - (1.5 + np.log(len(allowed)))) < TOL
    d.close()


def test_step_decode_logprobs_need_lse():
    w = workload(2)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    states, _ = w.initial_configs(batch=4)
    V = w.vocab.n_tokens
    lg = dev(w.logits(3, batch=4).view(np.int16))
    mask = torch.empty((4, d.info()["n_words"]), dtype=torch.int32, device="cuda")
    arg = torch.empty(4, dtype=torch.int32, device="cuda")
    lp = torch.empty((4, V), dtype=torch.float32, device="cuda")
    with pytest.raises(B.DominoError):
        B.domino_step_decode(d.h, dev(states), None, 4, lg.data_ptr(), B.DTYPE_BF16, V, mask, arg, None, lp)
    d.close()


@pytest.mark.parametrize("config", [1, 2, 3, 5])
def test_step_decode_with_update_matches_oracle(config):
    """states_out given: the merge advances each row by its argmax in place
    (config 1, fp32 logits: the separate kernels, then domino_advance)."""
    import oracle
    w = workload(config)
    P = oracle.Problem.from_workload(w)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    states, stacks = w.initial_configs()
    has_stack = w.automaton.rules is not None
    lg = w.logits(11)
    t = torch.from_numpy(lg.view(np.int16) if lg.dtype == np.uint16 else lg).cuda()
    dt = B.DTYPE_BF16 if lg.dtype == np.uint16 else B.DTYPE_F32
    V, b = w.vocab.n_tokens, len(states)
    st = dev(states)
    sk = dev(stacks.view(np.int64)) if has_stack else None
    mask = poison.empty((b, d.info()["n_words"]), torch.int32)
    arg = poison.empty(b, torch.int32)
    lse = poison.empty(b, torch.float32)
    B.domino_step_decode(d.h, st, sk, b, t.data_ptr(), dt, V, mask, arg, lse, None, st, sk)
    torch.cuda.synchronize()
    m_o, _, _ = P.step_mask(states, stacks if has_stack else None, n_threads=NT)
    a_o, l_o, _ = oracle.mask_logits(lg, m_o, n_threads=NT)
    s_o, k_o, bad = P.advance(states, stacks if has_stack else None, a_o, w.automaton.start)
    assert bad == 0
    assert_exact(mask, m_o, "mask")
    assert_exact(arg, np.asarray(a_o, np.int32), "argmax")
    assert_no_poison(lse, "lse")
    fin = np.isfinite(l_o)
    assert np.abs(lse.cpu().numpy()[fin] - l_o[fin]).max(initial=0) < TOL
    assert_exact(st, s_o, "states")
    if has_stack:
        assert_exact(sk, k_o, "stacks")
    assert d.device_error() == 0
    d.close()
