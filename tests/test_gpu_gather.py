"""The masked decode over bf16 logits when the batch has more rows than the GPU
has SMs (one CTA per row, compacted gathers of the allowed 16-byte logit
vectors), against the oracle: argmax and draws bit-exact, lse and log-probs
within 1e-3.  Rows mix every density the gather treats differently (nothing
allowed, one token, sparse vectors, vectors with three or more allowed tokens,
fully allowed rows), ties across vectors and warps, the row's last partial
vector, mask rows that do not start on 16-byte boundaries, padded row strides
and spans that take several load rounds.  Output buffers start as 0xAB bytes
(tests/poison.py)."""
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


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


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


def many_rows():
    return 2 * torch.cuda.get_device_properties(0).multi_processor_count + 9


def case(V, stride, seed):
    """bf16 logits [B][stride] and a mask [B][W] whose rows cycle through the
    densities and special cases."""
    rng = np.random.default_rng(seed)
    B_ = many_rows()
    x = (rng.standard_normal((B_, stride)) * 2.5).astype(np.float32)
    bits = np.zeros((B_, V), bool)
    for r in range(B_):
        k = r % 9
        if k == 0:
            pass                                          # nothing allowed
        elif k == 1:
            bits[r, rng.integers(V)] = True               # one token
        elif k == 2:
            bits[r] = rng.random(V) < 0.01                # sparse
        elif k == 3:
            bits[r] = rng.random(V) < 0.5                 # many vectors with 3+ tokens
        elif k == 4:
            bits[r] = True                                # everything
        elif k == 5:
            bits[r] = rng.random(V) < 0.9
            bits[r, V - 1] = True                         # the last (partial) vector
            x[r, V - 1] = 40.0                            # ... holds the maximum
        elif k == 6:
            # equal maxima in different vectors and warps: lowest id wins
            idx = np.sort(rng.choice(V, 6, replace=False))
            bits[r] = rng.random(V) < 0.2
            bits[r, idx] = True
            x[r, idx] = 30.0
        elif k == 7:
            # a larger logit masked out next to the allowed maximum
            bits[r] = rng.random(V) < 0.05
            j = int(rng.integers(1, V))
            bits[r, j - 1] = False
            x[r, j - 1] = 60.0
        else:
            bits[r, : min(V, 3000)] = True                # one dense block, rest empty
    xb = synth.f32_to_bf16_bits(x)
    return xb, packed(bits), B_


@pytest.mark.parametrize("V,stride", [(10003, 10008), (4104, 4104), (32768, 32768), (131077, 131080)])
def test_gather_matches_oracle(V, stride):
    import oracle
    assert stride % 8 == 0   # rows on 16-byte boundaries: the gather's precondition
    xb, m, B_ = case(V, stride, V)
    arg_o, lse_o, lp_o = oracle.mask_logits(xb, m, n_tokens=V, want_logprobs=True, n_threads=NT)
    d = vocab_handle(V)
    lg = dev(xb.view(np.int16)).view(torch.bfloat16)
    md = dev(m.view(np.int32))
    for want_lse, want_lp in ((False, False), (True, False), (True, True)):
        argmax = poison.empty(B_, torch.int32)
        lse = poison.empty(B_, torch.float32) if want_lse else None
        lp = poison.empty((B_, V), torch.float32) if want_lp else None
        B.domino_mask_logits(d.h, lg.data_ptr(), B.DTYPE_BF16, B_, stride, md, argmax, lse, lp)
        assert_exact(argmax, np.asarray(arg_o, np.int32), "argmax")
        if lse is not None:
            assert_no_poison(lse, "lse")
            g = lse.cpu().numpy().astype(np.float64)
            fin = np.isfinite(lse_o)
            assert (np.isfinite(g) == fin).all()
            assert np.abs(g[fin] - lse_o[fin]).max(initial=0) < TOL
        if lp is not None:
            assert_no_poison(lp, "log-probs")
            g = lp.cpu().numpy().astype(np.float64)
            fin = np.isfinite(lp_o)
            assert (np.isfinite(g) == fin).all()
            assert np.abs(g[fin] - lp_o[fin]).max(initial=0) < TOL
    assert arg_o[0] == -1
    assert d.device_error() == 0
    d.close()


@pytest.mark.parametrize("V,stride,temperature", [(10003, 10008, 0.8), (131077, 131080, 1.0)])
def test_gather_sample_matches_oracle(V, stride, temperature):
    import oracle
    xb, m, B_ = case(V, stride, V + 11)
    want = oracle.mask_sample(xb, m, temperature, 1234, 77, n_tokens=V, n_threads=NT)
    d = vocab_handle(V)
    lg = dev(xb.view(np.int16)).view(torch.bfloat16)
    tok = poison.empty(B_, torch.int32)
    B.domino_mask_sample(d.h, lg.data_ptr(), B.DTYPE_BF16, B_, stride, dev(m.view(np.int32)), temperature, 1234, 77,
                         tok)
    assert_exact(tok, np.asarray(want, np.int32), "draws")
    assert int(tok[0]) == -1
    d.close()


def test_gather_unaligned_mask_rows():
    """W odd: every other mask row starts off a 16-byte boundary."""
    import oracle
    V = 4000              # W = 125
    assert ((V + 31) // 32) % 2 == 1
    xb, m, B_ = case(V, V, 5)
    arg_o, lse_o, _ = oracle.mask_logits(xb, m, n_tokens=V, n_threads=NT)
    d = vocab_handle(V)
    argmax = poison.empty(B_, torch.int32)
    lse = poison.empty(B_, torch.float32)
    B.domino_mask_logits(d.h, dev(xb.view(np.int16)).view(torch.bfloat16).data_ptr(), B.DTYPE_BF16, B_, V,
                         dev(m.view(np.int32)), argmax, lse, None)
    assert_exact(argmax, np.asarray(arg_o, np.int32), "argmax")
    g = lse.cpu().numpy().astype(np.float64)
    fin = np.isfinite(lse_o)
    assert (np.isfinite(g) == fin).all()
    assert np.abs(g[fin] - lse_o[fin]).max(initial=0) < TOL
    d.close()
