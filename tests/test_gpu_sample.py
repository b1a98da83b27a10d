"""Sampling decode (Gumbel-max, Philox4x32-10 uniforms) through the C ABI
against the oracle's draw: tokens bit-exact on the same logits, masks, seed and
offset.  Masks fed to both sides come from the oracle.  Output buffers start
as 0xAB bytes (tests/poison.py)."""
import functools
import os

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

from paper_2403_06988_gb300 import Domino, synth  # noqa: E402
from paper_2403_06988_gb300 import _binding as B  # noqa: E402
import poison  # noqa: E402
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


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def logits_tensor(x):
    return dev(x.view(np.int16)).view(torch.bfloat16) if x.dtype == np.uint16 else dev(x)


def packed(bits):
    B_, V = bits.shape
    W = (V + 31) // 32
    p = np.zeros((B_, W * 32), np.uint8)
    p[:, :V] = bits
    return np.packbits(p, axis=1, bitorder="little").view("<u4")


def vocab_handle(V):
    d = Domino(0)
    d.load_vocab(synth.Vocab.from_tokens([bytes([i % 256]) for i in range(V)]))
    return d


@pytest.mark.parametrize("config,temperature,seed,offset", [
    (1, 1.0, 7, 0), (2, 0.7, 0x0123456789ABCDEF, 5), (3, 1.0, 42, (1 << 32) + 3), (5, 1.3, 2 ** 64 - 1, 17)])
def test_sample_matches_oracle_on_workloads(config, temperature, seed, offset):
    import oracle
    w = workload(config)
    P = oracle.Problem.from_workload(w)
    states, stacks = w.initial_configs()
    m, _, _ = P.step_mask(states, stacks if w.automaton.rules is not None else None, n_threads=NT)
    lg = w.logits(offset % 97)
    want = oracle.mask_sample(lg, m, temperature, seed, offset, n_threads=NT)
    d = Domino.from_parts(w.automaton, w.vocab, device=0)
    got = d.mask_sample(logits_tensor(lg), dev(m.view(np.int32)), temperature, seed, offset)
    assert_exact(got, np.asarray(want, np.int32), "draws")
    greedy, _, _ = oracle.mask_logits(lg, m)
    assert ((want >= 0) == (greedy >= 0)).all()
    d.close()


@pytest.mark.parametrize("V,stride,dtype", [(1000, 1000, "f32"), (1003, 1009, "bf16"), (65541, 65541, "bf16"),
                                            (777, 781, "f32")])
def test_sample_ragged_and_unaligned(V, stride, dtype):
    import oracle
    d = vocab_handle(V)
    rng = np.random.default_rng(V + 1)
    B_ = 6
    x = (rng.standard_normal((B_, stride)) * 3).astype(np.float32)
    if dtype == "bf16":
        x = synth.f32_to_bf16_bits(x)
    bits = rng.random((B_, V)) < 0.4
    bits[0] = False
    m = packed(bits)
    want = oracle.mask_sample(x, m, 0.9, 99, 3, n_tokens=V)
    tok = poison.empty(B_, torch.int32)
    lg = logits_tensor(x)   # held across the call: nothing else may reuse its memory
    B.domino_mask_sample(d.h, lg.data_ptr(), B.DTYPE_BF16 if dtype == "bf16" else B.DTYPE_F32, B_,
                         stride, dev(m.view(np.int32)), 0.9, 99, 3, tok)
    assert_exact(tok, np.asarray(want, np.int32), "draws")
    assert int(tok[0]) == -1
    d.close()


def test_sample_rows_beyond_one_pass_use_their_own_counter():
    import oracle
    V, B_ = 64, 4100
    d = vocab_handle(V)
    x = np.zeros((B_, V), np.float32)                 # uniform: the draw is decided by the counter alone
    m = packed(np.ones((B_, V), bool))
    want = oracle.mask_sample(x, m, 1.0, 5, 6, n_threads=NT)
    got = d.mask_sample(dev(x), dev(m.view(np.int32)), 1.0, 5, 6)
    assert_exact(got, np.asarray(want, np.int32), "draws")
    d.close()


@pytest.mark.parametrize("temperature", [0.0, -1.0, float("inf"), float("nan"), 1e-45])
def test_sample_rejects_bad_temperatures(temperature):
    d = vocab_handle(64)
    x = torch.zeros((2, 64), dtype=torch.float32, device="cuda")
    m = torch.zeros((2, 2), dtype=torch.int32, device="cuda")
    tok = torch.empty(2, dtype=torch.int32, device="cuda")
    with pytest.raises(B.DominoError) as e:
        B.domino_mask_sample(d.h, x, B.DTYPE_F32, 2, 64, m, temperature, 1, 0, tok)
    assert e.value.status == -1
    d.close()
