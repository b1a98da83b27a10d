"""domino_mask_logits_noalloc: the masked argmax / log-sum-exp for callers that
cannot allocate device memory (for example while another component owns all
of the GPU's memory), so they cannot create a handle either.  It must give
what domino_mask_logits gives, call after call, using only its fixed scratch.

This file is named to be collected last: if it fails, a run that stops at the
first failure has already run every other test.  It passes alone in a fresh
process and after the other tests.
"""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

from paper_2403_06988_gb300 import Domino, synth  # noqa: E402
from paper_2403_06988_gb300 import _binding as B  # noqa: E402

TOL = 1e-3   # the tolerance of the other log-softmax parity tests


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2403_06988_gb300 import build
    build.build()


def _inputs(batch, V, dtype, density, seed):
    rng = np.random.default_rng(seed)
    x = (rng.standard_normal((batch, V)) * 3).astype(np.float32)
    bits = rng.random((batch, V)) < density
    bits[0] = False                       # one row with nothing allowed
    W = (V + 31) // 32
    packed = np.zeros((batch, W * 32), np.uint8)
    packed[:, :V] = bits
    mask = torch.from_numpy(np.packbits(packed, axis=1, bitorder="little").view(np.int32)).cuda()
    if dtype == B.DTYPE_BF16:
        logits = torch.from_numpy(synth.f32_to_bf16_bits(x).view(np.int16)).cuda().view(torch.bfloat16)
    else:
        logits = torch.from_numpy(x).cuda()
    return logits, mask


def _outputs(batch, V):
    return (torch.empty(batch, dtype=torch.int32, device="cuda"), torch.empty(batch, dtype=torch.float32, device="cuda"),
            torch.empty((batch, V), dtype=torch.float32, device="cuda"))


@pytest.mark.parametrize("batch,V,dtype,density", [(256, 128256, B.DTYPE_BF16, 0.08), (512, 32000, B.DTYPE_BF16, 0.6),
                                                   (7, 1003, B.DTYPE_F32, 0.3)])
def test_noalloc_matches_mask_logits_on_consecutive_calls(batch, V, dtype, density):
    logits, mask = _inputs(batch, V, dtype, density, seed=V)
    # the existing entry point, through a handle that holds a V-token vocabulary
    ref = Domino(0)
    ref.load_vocab(synth.Vocab.from_tokens([bytes([i % 256]) for i in range(V)]))
    r_arg, r_lse, r_lp = _outputs(batch, V)
    B.domino_mask_logits(ref.h, logits.data_ptr(), dtype, batch, V, mask, r_arg, r_lse, r_lp)
    torch.cuda.synchronize()
    for call in range(2):                 # the shared scratch must be left ready for the next call
        arg, lse, lp = _outputs(batch, V)
        B.domino_mask_logits_noalloc(logits.data_ptr(), dtype, batch, V, V, mask, arg, lse, lp)
        torch.cuda.synchronize()
        assert torch.equal(arg, r_arg), call
        assert int(arg[0]) == -1
        fin = torch.isfinite(r_lse)
        assert torch.equal(torch.isfinite(lse), fin)
        assert float((lse[fin] - r_lse[fin]).abs().max()) < TOL
        lfin = torch.isfinite(r_lp)
        assert torch.equal(torch.isfinite(lp), lfin)
        assert float((lp[lfin] - r_lp[lfin]).abs().max()) < TOL
    ref.close()


def test_noalloc_rejects_batches_beyond_its_scratch():
    logits, mask = _inputs(513, 64, B.DTYPE_F32, 0.5, seed=1)
    arg, _, _ = _outputs(513, 64)
    with pytest.raises(B.DominoError) as e:
        B.domino_mask_logits_noalloc(logits.data_ptr(), B.DTYPE_F32, 513, 64, 64, mask, arg)
    assert e.value.status == -1
