"""domino_mask_logits_noalloc: the masked argmax / log-sum-exp for callers that
cannot allocate device memory (for example while another component owns all
of the GPU's memory), so they cannot create a handle either.  Call after
call, using only its fixed scratch, it must give the oracle's masked argmax
(bit-exact) and log-sum-exp and log-probs (within 1e-3), and what
domino_mask_logits gives.  Output buffers start as 0xAB bytes.

This file is named to be collected last: if it fails, a run that stops at the
first failure has already run every other test.  It passes alone in a fresh
process and after the other tests.
"""
import os

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

from paper_2403_06988_gb300 import Domino, synth  # noqa: E402
from paper_2403_06988_gb300 import _binding as B  # noqa: E402
import poison  # noqa: E402
from poison import assert_exact, assert_no_poison  # noqa: E402

TOL = 1e-3   # the tolerance of the other log-softmax parity tests


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2403_06988_gb300 import build
    build.build()


def _inputs(batch, V, dtype, density, seed):
    """Host logits (float32, or bf16 bits as uint16) and packed masks, and
    their device copies."""
    rng = np.random.default_rng(seed)
    x = (rng.standard_normal((batch, V)) * 3).astype(np.float32)
    bits = rng.random((batch, V)) < density
    bits[0] = False                       # one row with nothing allowed
    W = (V + 31) // 32
    packed = np.zeros((batch, W * 32), np.uint8)
    packed[:, :V] = bits
    m = np.packbits(packed, axis=1, bitorder="little").view("<u4")
    mask = torch.from_numpy(m.view(np.int32)).cuda()
    if dtype == B.DTYPE_BF16:
        x = synth.f32_to_bf16_bits(x)
        logits = torch.from_numpy(x.view(np.int16)).cuda().view(torch.bfloat16)
    else:
        logits = torch.from_numpy(x).cuda()
    return x, m, logits, mask


def _outputs(batch, V):
    return (poison.empty(batch, torch.int32), poison.empty(batch, torch.float32),
            poison.empty((batch, V), torch.float32))


def _close(got, want, what):
    """got (device, fp32) within TOL of want (float64, host); -inf where want is."""
    assert_no_poison(got, what)
    g = got.cpu().numpy().astype(np.float64)
    fin = np.isfinite(want)
    assert (np.isfinite(g) == fin).all(), what
    assert (g[~fin] == -np.inf).all(), what
    assert np.abs(g[fin] - want[fin]).max(initial=0) < TOL, what


@pytest.mark.parametrize("batch,V,dtype,density", [(256, 128256, B.DTYPE_BF16, 0.08), (512, 32000, B.DTYPE_BF16, 0.6),
                                                   (7, 1003, B.DTYPE_F32, 0.3)])
def test_noalloc_matches_oracle_and_mask_logits_on_consecutive_calls(batch, V, dtype, density):
    import oracle
    x, m, logits, mask = _inputs(batch, V, dtype, density, seed=V)
    a_o, l_o, lp_o = oracle.mask_logits(x, m, want_logprobs=True, n_threads=os.cpu_count() or 1)
    assert a_o[0] == -1
    # the handle's entry point on the same inputs
    ref = Domino(0)
    ref.load_vocab(synth.Vocab.from_tokens([bytes([i % 256]) for i in range(V)]))
    r_arg, r_lse, r_lp = _outputs(batch, V)
    B.domino_mask_logits(ref.h, logits.data_ptr(), dtype, batch, V, mask, r_arg, r_lse, r_lp)
    torch.cuda.synchronize()
    for call in range(2):                 # the shared scratch must be left ready for the next call
        arg, lse, lp = _outputs(batch, V)
        B.domino_mask_logits_noalloc(logits.data_ptr(), dtype, batch, V, V, mask, arg, lse, lp)
        torch.cuda.synchronize()
        assert_exact(arg, a_o, f"argmax, call {call}")
        _close(lse, l_o, f"lse, call {call}")
        _close(lp, lp_o, f"log-probs, call {call}")
        assert torch.equal(arg, r_arg), call
        fin = torch.isfinite(r_lse)
        assert float((lse[fin] - r_lse[fin]).abs().max()) < TOL
        lfin = torch.isfinite(r_lp)
        assert float((lp[lfin] - r_lp[lfin]).abs().max()) < TOL
    ref.close()


def test_noalloc_rejects_batches_beyond_its_scratch():
    _, _, logits, mask = _inputs(513, 64, B.DTYPE_F32, 0.5, seed=1)
    arg, _, _ = _outputs(513, 64)
    with pytest.raises(B.DominoError) as e:
        B.domino_mask_logits_noalloc(logits.data_ptr(), B.DTYPE_F32, 513, 64, 64, mask, arg)
    assert e.value.status == -1
