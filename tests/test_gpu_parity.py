"""GPU parity: libdomino.so (through its C ABI) against the CPU oracle.

Masks, next states, argmax, advanced configurations: bit-exact.
lse and log-probs: within 1e-3 absolute (fp32 accumulation of bf16/fp32
inputs against the oracle's float64).
Every output buffer starts filled with 0xAB bytes (tests/poison.py), so a
word a kernel leaves unwritten fails the comparison.
"""
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
DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2403_06988_gb300 import build
    build.build()
    torch.cuda.init()


@functools.lru_cache(maxsize=None)
def workload(config):
    return synth.workload(config)


@functools.lru_cache(maxsize=None)
def configs(config, batch=None):
    return workload(config).initial_configs(batch=batch)


@functools.lru_cache(maxsize=None)
def handle(config):
    w = workload(config)
    return Domino.from_parts(w.automaton, w.vocab, device=0)


@functools.lru_cache(maxsize=None)
def problem(config):
    import oracle
    return oracle.Problem.from_workload(workload(config))


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def u32(t):
    return t.cpu().numpy().view(np.uint32)


def logits_tensor(np_logits):
    if np_logits.dtype == np.uint16:
        return dev(np_logits.view(np.int16)).view(torch.bfloat16)
    return dev(np_logits)


def assert_logits_match(arg_g, lse_g, lp_g, arg_o, lse_o, lp_o):
    assert_exact(arg_g, np.asarray(arg_o, np.int32), "argmax")
    if lse_g is not None:
        assert_no_poison(lse_g, "lse")
        lg = lse_g.cpu().numpy().astype(np.float64)
        fin = np.isfinite(lse_o)
        assert (np.isfinite(lg) == fin).all()
        assert np.abs(lg[fin] - lse_o[fin]).max(initial=0) < TOL
    if lp_g is not None:
        assert_no_poison(lp_g, "log-probs")
        pg = lp_g.cpu().numpy().astype(np.float64)
        fin = np.isfinite(lp_o)
        assert (np.isfinite(pg) == fin).all()
        assert (pg[~fin] == -np.inf).all()
        assert np.abs(pg[fin] - lp_o[fin]).max(initial=0) < TOL


# --------------------------------------------------------------------------
# step_mask
# --------------------------------------------------------------------------
@pytest.mark.parametrize("config", [1, 2, 3, 5])
def test_step_mask_parity(config):
    w = workload(config)
    states, stacks = configs(config)
    d = handle(config)
    # the walk chosen from the automaton: the prefix tree unless states loop
    # on many classes (configs 2 and 5: strings); tests/test_gpu_tree_walk.py
    # and tests/test_gpu_token_walk.py force each walk
    if config in (3, 5):
        assert d.info()["walk_tree"] == (1 if config == 3 else 0)
    st = dev(states)
    sk = dev(stacks.view(np.int64)) if w.automaton.rules is not None else None
    mask, nxt = d.step_mask(st, sk, want_next=True)
    mask2, _ = d.step_mask(st, sk, want_next=False)
    torch.cuda.synchronize()
    m_o, n_o, bad = problem(config).step_mask(states, stacks if sk is not None else None, want_next=True,
                                              n_threads=NT)
    assert bad == 0
    assert_exact(mask, m_o, "mask")
    assert_exact(mask2, m_o, "mask (no next states)")
    assert_exact(nxt, n_o, "next")
    assert d.device_error() == 0


def test_step_mask_depth32_rows():
    """Config-5 rows at the maximum depth: every push must be rejected."""
    w = workload(5)
    extra_s, extra_k = [], []
    rng = np.random.default_rng(9)
    while len(extra_s) < 16:
        s, stk = synth.random_pda_walk(w.automaton, rng, 32)
        if len(stk) == 32:
            extra_s.append(s)
            extra_k.append(synth.pack_stack(stk))
    st = np.array(extra_s, np.int32)
    sk = np.array(extra_k, np.uint64)
    d = handle(5)
    mask, nxt = d.step_mask(dev(st), dev(sk.view(np.int64)), want_next=True)
    m_o, n_o, bad = problem(5).step_mask(st, sk, want_next=True, n_threads=NT)
    assert bad == 0
    assert_exact(mask, m_o, "mask")
    assert_exact(nxt, n_o, "next")
    toks = w.vocab.tokens()
    lb = toks.index(b"{")
    push_states = {int(r["state"]) for r in w.automaton.rules if r["kind"] == synth.RULE_PUSH}
    pushing = [i for i in range(len(st)) if int(st[i]) in push_states]
    assert not any((m_o[i, lb >> 5] >> (lb & 31)) & 1 for i in pushing)


# --------------------------------------------------------------------------
# mask_logits
# --------------------------------------------------------------------------
@pytest.mark.parametrize("config", [1, 2, 3, 5])
def test_mask_logits_parity(config):
    import oracle
    w = workload(config)
    states, stacks = configs(config)
    m_o, _, _ = problem(config).step_mask(states, stacks if w.automaton.rules is not None else None, n_threads=NT)
    lg = w.logits(0)
    arg_o, lse_o, lp_o = oracle.mask_logits(lg, m_o, want_logprobs=True, n_threads=NT)
    d = handle(config)
    for want_lp in (False, True):
        arg, lse, lp = d.mask_logits(logits_tensor(lg), dev(m_o.view(np.int32)), want_lse=True,
                                     want_logprobs=want_lp)
        assert_logits_match(arg, lse, lp, arg_o, lse_o, lp_o if want_lp else None)


def test_mask_logits_edge_rows():
    import oracle
    d = handle(2)
    V = workload(2).vocab.n_tokens
    W = (V + 31) // 32
    rng = np.random.default_rng(21)
    B_ = 6
    x = synth.f32_to_bf16_bits((rng.standard_normal((B_, V)) * 2).astype(np.float32))
    bits = np.zeros((B_, V), bool)
    # row 0 all masked; row 1 one token; row 2 ties at the max (lowest id wins);
    # row 3 larger masked logits; row 4 last token only; row 5 dense
    bits[1, 12345] = True
    x[2, [100, 5000, 31000]] = synth.f32_to_bf16_bits(np.array([9.0], np.float32))[0]
    bits[2, [100, 5000, 31000, 7]] = True
    x[3, 0] = synth.f32_to_bf16_bits(np.array([50.0], np.float32))[0]
    bits[3, 1:200] = True
    bits[4, V - 1] = True
    bits[5] = rng.random(V) < 0.7
    packed = np.zeros((B_, W * 32), np.uint8)
    packed[:, :V] = bits
    m = np.packbits(packed, axis=1, bitorder="little").view("<u4")
    arg_o, lse_o, lp_o = oracle.mask_logits(x, m, want_logprobs=True)
    arg, lse, lp = d.mask_logits(logits_tensor(x), dev(m.view(np.int32)), want_lse=True, want_logprobs=True)
    assert arg_o[0] == -1 and arg_o[2] == 100
    assert_logits_match(arg, lse, lp, arg_o, lse_o, lp_o)


@pytest.mark.parametrize("V,stride,dtype", [(1000, 1000, "f32"), (1003, 1009, "bf16"), (4099, 4099, "f32"),
                                            (777, 781, "f32"), (65541, 65541, "bf16")])
def test_mask_logits_ragged_and_unaligned(V, stride, dtype):
    """V not a multiple of 8/32, odd row strides (scalar path), several chunks."""
    import oracle
    d = vocab_handle(V)
    rng = np.random.default_rng(V)
    B_ = 5
    x = (rng.standard_normal((B_, stride)) * 3).astype(np.float32)
    if dtype == "bf16":
        x = synth.f32_to_bf16_bits(x)
    bits = rng.random((B_, V)) < 0.4
    bits[0] = False
    W = (V + 31) // 32
    packed = np.zeros((B_, W * 32), np.uint8)
    packed[:, :V] = bits
    m = np.packbits(packed, axis=1, bitorder="little").view("<u4")
    arg_o, lse_o, lp_o = oracle.mask_logits(x, m, n_tokens=V, want_logprobs=True)
    xt = logits_tensor(x)
    argmax = poison.empty(B_, torch.int32, DEV)
    lse = poison.empty(B_, torch.float32, DEV)
    lp = poison.empty((B_, V), torch.float32, DEV)
    B.domino_mask_logits(d.h, xt.data_ptr(), B.DTYPE_BF16 if dtype == "bf16" else B.DTYPE_F32, B_, stride,
                         dev(m.view(np.int32)), argmax, lse, lp)
    assert_logits_match(argmax, lse, lp, arg_o, lse_o, lp_o)


def vocab_handle(V):
    """A handle holding only a V-token vocabulary (enough for mask_logits)."""
    d = Domino(0)
    d.load_vocab(synth.Vocab.from_tokens([bytes([i % 256]) for i in range(V)]))
    return d


def test_mask_logits_more_rows_than_one_pass():
    import oracle
    d = handle(1)
    V = 1024
    B_ = 4100
    rng = np.random.default_rng(5)
    x = rng.standard_normal((B_, V)).astype(np.float32)
    bits = rng.random((B_, V)) < 0.1
    m = np.packbits(bits, axis=1, bitorder="little").view("<u4")
    arg_o, lse_o, _ = oracle.mask_logits(x, m, n_threads=NT)
    arg, lse, _ = d.mask_logits(dev(x), dev(m.view(np.int32)), want_lse=True)
    assert_logits_match(arg, lse, None, arg_o, lse_o, None)


# --------------------------------------------------------------------------
# advance and the decode loop
# --------------------------------------------------------------------------
@pytest.mark.parametrize("config", [1, 2, 3, 5])
def test_advance_parity(config):
    w = workload(config)
    states, stacks = configs(config)
    has_stack = w.automaton.rules is not None
    rng = np.random.default_rng(config)
    Bn = len(states)
    tokens = rng.integers(0, w.vocab.n_tokens, size=Bn).astype(np.int32)
    tokens[::7] = -1
    tokens[1::7] = w.vocab.eos_id
    # half of the rows take an allowed token (the oracle's argmax of random logits)
    import oracle
    m_o, _, _ = problem(config).step_mask(states, stacks if has_stack else None, n_threads=NT)
    arg_o, _, _ = oracle.mask_logits(w.logits(1), m_o)
    tokens[2::2] = arg_o[2::2]
    so_o, wo_o, bad = problem(config).advance(states, stacks if has_stack else None, tokens, w.automaton.start)
    assert bad == 0
    d = handle(config)
    st = dev(states)
    sk = dev(stacks.view(np.int64)) if has_stack else None
    so = poison.empty_like(st)
    wo = poison.empty_like(sk) if has_stack else None
    d.advance(st, sk, dev(tokens), states_out=so, stacks_out=wo)
    assert_exact(so, so_o, "states")
    if has_stack:
        assert_exact(wo, wo_o, "stacks")
    # in place
    d.advance(st, sk, dev(tokens))
    assert_exact(st, so_o, "states in place")


@pytest.mark.parametrize("config,steps", [(1, 64), (2, 40), (5, 12)])
def test_decode_loop_parity(config, steps):
    """Alg. 1 end to end: mask -> masked argmax -> update, compared each step."""
    import oracle
    w = workload(config)
    states, stacks = configs(config)
    has_stack = w.automaton.rules is not None
    d = handle(config)
    st = dev(states)
    sk = dev(stacks.view(np.int64)) if has_stack else None
    s_o, k_o = states.copy(), stacks.copy()
    for i in range(steps):
        lg = w.logits(i)
        mask, _ = d.step_mask(st, sk)
        arg, lse, _ = d.mask_logits(logits_tensor(lg), mask)
        d.advance(st, sk, arg)
        m_o, _, _ = problem(config).step_mask(s_o, k_o if has_stack else None, n_threads=NT)
        a_o, l_o, _ = oracle.mask_logits(lg, m_o)
        s_o, k_o, _ = problem(config).advance(s_o, k_o if has_stack else None, a_o, w.automaton.start)
        assert_exact(mask, m_o, f"mask, step {i}")
        assert_logits_match(arg, lse, None, a_o, l_o, None)
        assert (st.cpu().numpy() == s_o).all(), i
        if has_stack:
            assert (sk.cpu().numpy().view(np.uint64) == k_o).all(), i


@pytest.mark.parametrize("pinned", [False, True])
@pytest.mark.parametrize("config", [3, 5])
def test_decode_step_host_matches_oracle(config, pinned):
    """Pageable logits are copied in chunks of rows and each chunk is decoded as
    it lands; pinned logits are read in place.  Tokens, lse and the new
    configurations match the oracle either way."""
    import oracle
    w = workload(config)
    states, stacks = configs(config)
    has_stack = w.automaton.rules is not None
    d = handle(config)
    lg = w.logits(5)
    if pinned:
        lg = torch.from_numpy(lg.view(np.int16) if lg.dtype == np.uint16 else lg).pin_memory().numpy()
        lg = lg.view(np.uint16) if lg.dtype == np.int16 else lg
    s_host = states.copy()
    k_host = stacks.copy() if has_stack else None
    tok = poison.host(len(states), np.int32)
    lse_h = poison.host(len(states), np.float32)
    dt = B.DTYPE_BF16 if lg.dtype == np.uint16 else B.DTYPE_F32
    B.domino_decode_step_host(d.h, lg, dt, len(states), s_host, k_host, tok, lse_h, stream=0)
    P = problem(config)
    m, _, _ = P.step_mask(states, stacks if has_stack else None, n_threads=NT)
    a_o, l_o, _ = oracle.mask_logits(lg, m)
    s_o, k_o, _ = P.advance(states, stacks if has_stack else None, a_o, w.automaton.start)
    assert_exact(tok, a_o, "tokens")
    assert_no_poison(lse_h, "lse")
    fin = np.isfinite(l_o)
    assert np.abs(lse_h[fin] - l_o[fin]).max(initial=0) < TOL
    assert (s_host == s_o).all()
    if has_stack:
        assert (k_host == k_o).all()


@pytest.mark.parametrize("config", [2, 5])
def test_decode_step_host_replayed_steps_match_oracle(config):
    """On a non-default stream the host-buffer step is recorded once per set of
    buffers and replayed: a multi-step loop over two alternating pinned logits
    buffers and one pageable one gives the oracle's tokens and configurations
    every step."""
    import oracle
    w = workload(config)
    has_stack = w.automaton.rules is not None
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    P = problem(config)
    states, stacks = w.initial_configs()
    s_host = torch.from_numpy(states.copy()).pin_memory()
    k_host = torch.from_numpy(stacks.view(np.int64).copy()).pin_memory() if has_stack else None
    tok = poison.empty(len(states), torch.int32, pin=True)
    lse_h = poison.empty(len(states), torch.float32, pin=True)
    bufs = [torch.from_numpy(w.logits(40 + i).view(np.int16)).pin_memory() for i in range(2)]
    bufs.append(torch.from_numpy(w.logits(42).view(np.int16)))          # pageable: the copy path
    s_o, k_o = states.copy(), stacks.copy()
    st = torch.cuda.Stream()
    for i in range(7):
        b = bufs[i % 3]
        tok.view(torch.uint8).fill_(poison.POISON_BYTE)
        lse_h.view(torch.uint8).fill_(poison.POISON_BYTE)
        B.domino_decode_step_host(d.h, b.data_ptr(), B.DTYPE_BF16, len(states), s_host.data_ptr(),
                                  k_host.data_ptr() if has_stack else None, tok.data_ptr(), lse_h.data_ptr(),
                                  stream=st.cuda_stream)
        lg = b.numpy().view(np.uint16)
        m, _, _ = P.step_mask(s_o, k_o if has_stack else None, n_threads=NT)
        a_o, l_o, _ = oracle.mask_logits(lg, m)
        s_o, k_o2, _ = P.advance(s_o, k_o if has_stack else None, a_o, w.automaton.start)
        k_o = k_o2 if has_stack else k_o
        assert_exact(tok, a_o, f"tokens, step {i}")
        assert_no_poison(lse_h, f"lse, step {i}")
        fin = np.isfinite(l_o)
        assert np.abs(lse_h.numpy()[fin] - l_o[fin]).max(initial=0) < TOL
        assert (s_host.numpy() == s_o).all(), i
        if has_stack:
            assert (k_host.numpy().view(np.uint64) == k_o).all(), i
    assert d.device_error() == 0
    d.close()


def test_decode_step_host_path_choice_keeps_results():
    """Pinned bf16 logits: the handle times the in-place and the copy path on
    its own calls, uses the faster and retimes the other every 64th call; 70
    replayed steps cover both paths and the switch, every step equal to the
    oracle."""
    import oracle
    w = workload(2)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    P = problem(2)
    states, _ = w.initial_configs()
    s_host = torch.from_numpy(states.copy()).pin_memory()
    tok = poison.empty(len(states), torch.int32, pin=True)
    lse_h = poison.empty(len(states), torch.float32, pin=True)
    bufs = [torch.from_numpy(w.logits(60 + i).view(np.int16)).pin_memory() for i in range(2)]
    s_o = states.copy()
    st = torch.cuda.Stream()
    for i in range(70):
        b = bufs[i % 2]
        tok.view(torch.uint8).fill_(poison.POISON_BYTE)
        lse_h.view(torch.uint8).fill_(poison.POISON_BYTE)
        B.domino_decode_step_host(d.h, b.data_ptr(), B.DTYPE_BF16, len(states), s_host.data_ptr(), None,
                                  tok.data_ptr(), lse_h.data_ptr(), stream=st.cuda_stream)
        m, _, _ = P.step_mask(s_o, None, n_threads=NT)
        a_o, l_o, _ = oracle.mask_logits(b.numpy().view(np.uint16), m)
        s_o, _, _ = P.advance(s_o, None, a_o, w.automaton.start)
        assert_exact(tok, a_o, f"tokens, step {i}")
        assert_no_poison(lse_h, f"lse, step {i}")
        fin = np.isfinite(l_o)
        assert np.abs(lse_h.numpy()[fin] - l_o[fin]).max(initial=0) < TOL, i
        assert (s_host.numpy() == s_o).all(), i
    assert d.device_error() == 0
    d.close()


def test_decode_step_host_batch_grows_on_a_recording_stream():
    """Pinned bf16 logits on a non-default stream, with batches growing from
    call to call.  On a fresh handle the first calls take the in-place path
    (it has not been timed yet), and from the third call on a step is recorded
    into a CUDA graph: the fused decode's per-window partials must have grown
    before that recording starts.  Three calls at one batch, then larger
    batches, every call equal to the oracle."""
    import oracle
    w = workload(2)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    P = problem(2)
    st = torch.cuda.Stream()
    plan = [8, 16, 32, 32, 32, 32, 64, 64, 96]
    big = max(plan)
    rng = np.random.default_rng(123)
    live = np.nonzero(w.automaton.live)[0]
    s_all = rng.choice(live, size=big).astype(np.int32)
    lg_all = torch.from_numpy(w.logits(70, batch=big).view(np.int16)).pin_memory()
    s_host = torch.from_numpy(s_all.copy()).pin_memory()
    tok = poison.empty(big, torch.int32, pin=True)
    lse_h = poison.empty(big, torch.float32, pin=True)
    s_o = s_all.copy()
    for i, b in enumerate(plan):
        tok.view(torch.uint8).fill_(poison.POISON_BYTE)
        lse_h.view(torch.uint8).fill_(poison.POISON_BYTE)
        before = s_o[:b].copy()
        B.domino_decode_step_host(d.h, lg_all.data_ptr(), B.DTYPE_BF16, b, s_host.data_ptr(), None, tok.data_ptr(),
                                  lse_h.data_ptr(), stream=st.cuda_stream)
        lg = lg_all.numpy().view(np.uint16)[:b]
        m, _, _ = P.step_mask(before, None, n_threads=NT)
        a_o, l_o, _ = oracle.mask_logits(lg, m)
        nxt, _, _ = P.advance(before, None, a_o, w.automaton.start)
        s_o[:b] = nxt
        assert_exact(tok[:b], a_o, f"tokens, call {i} (batch {b})")
        assert_no_poison(lse_h[:b], f"lse, call {i}")
        fin = np.isfinite(l_o)
        assert np.abs(lse_h.numpy()[:b][fin] - l_o[fin]).max(initial=0) < TOL, i
        assert (s_host.numpy() == s_o).all(), i
    assert d.device_error() == 0
    d.close()


def test_decode_step_host_matches_device_path():
    w = workload(2)
    states, _ = configs(2)
    d = handle(2)
    lg = w.logits(3)
    mask, _ = d.step_mask(dev(states))
    arg, lse, _ = d.mask_logits(logits_tensor(lg), mask)
    nxt = dev(states)
    d.advance(nxt, None, arg)
    s_host = states.copy()
    tok = poison.host(len(states), np.int32)
    lse_h = poison.host(len(states), np.float32)
    B.domino_decode_step_host(d.h, lg, B.DTYPE_BF16, len(states), s_host, None, tok, lse_h, stream=0)
    assert_no_poison(lse_h, "lse")
    assert (tok == arg.cpu().numpy()).all()
    assert (s_host == nxt.cpu().numpy()).all()
    assert np.abs(lse_h - lse.cpu().numpy()).max() < 1e-6


# --------------------------------------------------------------------------
# precompute
# --------------------------------------------------------------------------
def test_precompute_table_full_config2():
    w = workload(2)
    d = handle(2)
    nxt, mask = d.precompute_table()
    Q = w.automaton.n_states
    m_o, n_o, _ = problem(2).step_mask(np.arange(Q, dtype=np.int32), want_next=True, n_threads=NT)
    assert_exact(mask, m_o, "table mask")
    assert_exact(nxt, n_o, "table next")


def test_precompute_table_config4_full():
    """The full-size state x token table (Q = 20000, V = 128256, Alg. 2's
    traversal for every state): every row of mask and next states equal to the
    all-core oracle, compared in blocks of 2000 states; the table's invariants
    on the device; table row q == step_mask from q on sampled rows."""
    w = workload(4)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    assert d.info()["walk_tree"] == 1
    nxt, mask = d.precompute_table()
    torch.cuda.synchronize()
    Q, V = w.automaton.n_states, w.vocab.n_tokens
    assert nxt.shape == (Q, V)
    P = problem_c4()
    blk = 2000
    for q0 in range(0, Q, blk):
        q1 = min(Q, q0 + blk)
        m_o, n_o, bad = P.step_mask(np.arange(q0, q1, dtype=np.int32), want_next=True, n_threads=NT)
        assert bad == 0
        assert_exact(mask[q0:q1], m_o, f"table mask, states {q0}..{q1 - 1}")
        assert_exact(nxt[q0:q1], n_o, f"table next, states {q0}..{q1 - 1}")
        del m_o, n_o
    # invariants on the whole table, computed on the device
    tok = torch.arange(V, device=DEV)
    for q0 in range(0, Q, blk):
        blk_n = nxt[q0:q0 + blk]
        blk_m = mask[q0:q0 + blk]
        bit = (blk_m[:, tok >> 5] >> (tok & 31).to(torch.int32)) & 1
        assert torch.equal(bit == 1, blk_n != 0)
    assert int(mask[0].abs().sum()) == 0 and int(nxt[0].abs().sum()) == 0
    # table row q == step_mask from q
    rng = np.random.default_rng(44)
    rows = np.unique(np.concatenate([[0, 1, 2, Q - 1, 1999, 2000, 2001], rng.integers(0, Q, 57)])).astype(np.int32)
    sm, sn = d.step_mask(dev(rows), None, want_next=True)
    assert torch.equal(sm, mask[rows.tolist()]) and torch.equal(sn, nxt[rows.tolist()])
    del nxt, mask
    d.close()
    torch.cuda.empty_cache()


@functools.lru_cache(maxsize=None)
def problem_c4():
    import oracle
    return oracle.Problem.from_workload(workload(4))


def test_precompute_refuses_pushdown():
    with pytest.raises(B.DominoError) as e:
        handle(5).precompute_table()
    assert e.value.status == -3


# --------------------------------------------------------------------------
# tiny grammars, ragged vocabularies, invalid inputs
# --------------------------------------------------------------------------
def test_fig3_worked_example_on_gpu():
    a = synth.fig3_expr_pda()
    v = synth.fig3_vocab()
    d = Domino.from_parts(a, v, device=0)
    # configuration after "(12": state int_nonzero (2), one '(' on the stack
    mask, nxt = d.step_mask(dev(np.array([2], np.int32)), dev(np.array([synth.pack_stack([0])], np.int64)),
                            want_next=True)
    allowed = [b"0", b"1", b"2", b"12", b")", b"+", b"+1", b"1 +"]
    toks = v.tokens()
    want = np.zeros((1, (len(toks) + 31) // 32), np.uint32)
    for t, tok in enumerate(toks):
        if tok in allowed:
            want[0, t >> 5] |= np.uint32(1 << (t & 31))
    assert_exact(mask, want, "Fig. 3 mask after (12")


@pytest.mark.parametrize("name", ["dyck2", "int_regex", "dyck_ctx"])
def test_tiny_grammar_parity(name):
    import oracle
    a = {"dyck2": lambda: synth.dyck2_pda(3), "int_regex": synth.int_regex_dfa,
         "dyck_ctx": lambda: synth.dyck_ctx_pda(3)}[name]()
    alpha = {"dyck2": b"{}[]a", "int_regex": b"-0123", "dyck_ctx": b"{}[]abc"}[name]
    v = synth.all_strings_vocab(alpha, 4)
    d = Domino.from_parts(a, v, device=0)
    P = oracle.Problem.from_parts(a, v)
    # configurations: every live state with a few stacks
    states, stacks = [], []
    for q in range(1, a.n_states):
        for stk in ([], [0], [1], [1, 0], [0, 1, 1]):
            if len(stk) <= a.max_depth:
                states.append(q)
                stacks.append(synth.pack_stack(stk))
    states = np.array(states, np.int32)
    stacks = np.array(stacks, np.uint64)
    mask, nxt = d.step_mask(dev(states), dev(stacks.view(np.int64)), want_next=True)
    m_o, n_o, bad = P.step_mask(states, stacks, want_next=True)
    assert bad == 0
    assert_exact(mask, m_o, "mask")
    assert_exact(nxt, n_o, "next")


def test_ragged_vocab_long_tokens_eos_in_middle():
    """V % 1024 != 0, V % 4 != 0, tokens longer than 16 bytes, EOS not last,
    empty non-EOS token, pad bits of the last word."""
    import oracle
    a = synth.int_regex_dfa()
    rng = np.random.default_rng(8)
    toks = set()
    while len(toks) < 2500:
        L = int(rng.integers(1, 40))
        toks.add(rng.choice(np.frombuffer(b"-0123456789x", np.uint8), L).tobytes())
    toks = sorted(toks)
    toks.insert(700, b"")          # EOS
    toks.insert(1500, b"")         # an empty token that is not EOS
    v = synth.Vocab.from_tokens(toks, eos_id=700)
    assert v.n_tokens % 4 != 0 and v.n_tokens % 1024 != 0
    d = Domino.from_parts(a, v, device=0)
    P = oracle.Problem.from_parts(a, v)
    states = np.array([1, 2, 3, 4, 0, 1, 3], np.int32)
    mask, nxt = d.step_mask(dev(states), None, want_next=True)
    m_o, n_o, _ = P.step_mask(states, want_next=True)
    assert_exact(mask, m_o, "mask")
    assert_exact(nxt, n_o, "next")
    assert (u32(mask)[:, -1] >> (v.n_tokens % 32) == 0).all()


def test_invalid_inputs_set_error_word():
    w = workload(5)
    d = handle(5)
    assert d.device_error() == 0
    states = np.array([5, -1, 300, 7, 7, 7], np.int32)
    stacks = np.array([0, 0, 0, 33 << 32, (1 << 32) | 2, 1 << 41], np.uint64)
    mask, nxt = d.step_mask(dev(states), dev(stacks.view(np.int64)), want_next=True)
    m = u32(mask)
    assert (m[1:] == 0).all() and (nxt[1:] == 0).all()
    assert m[0].any()
    m_o, n_o, bad = problem(5).step_mask(states, stacks, want_next=True)
    assert bad == 5
    assert_exact(mask, m_o, "mask")
    assert_exact(nxt, n_o, "next")
    code = d.device_error()
    assert code == (B.DEVERR_BAD_STATE | B.DEVERR_BAD_STACK)
    assert d.device_error() == 0                      # cleared on read
    # advance: token id out of range
    st = dev(np.array([5, 5], np.int32))
    d.advance(st, dev(np.zeros(2, np.int64)), dev(np.array([w.vocab.n_tokens + 5, -1], np.int32)))
    assert st.cpu().numpy().tolist() == [0, w.automaton.start]
    assert d.device_error() == B.DEVERR_BAD_TOKEN


def test_zero_batch_is_noop_and_args_checked():
    d = handle(1)
    d.step_mask(dev(np.zeros(0, np.int32)))
    with pytest.raises(B.DominoError):
        B.domino_mask_logits(d.h, 0, 7, 1, 1024, 0, 0)        # bad dtype
    with pytest.raises(B.DominoError):
        B.domino_mask_logits(d.h, 0, 0, 1, 100, 0, 0)         # stride < V
