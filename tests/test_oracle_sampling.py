"""Pins of the oracle's sampling decode (Gumbel-max over the masked logits).

- Philox4x32-10 against the published known-answer vectors of its authors
  (Salmon et al., SC'11; counter, key -> output).
- The fp32 logarithm against math.log.
- The draw's distribution against softmax(x / T) of the allowed tokens
  (chi-square), masked tokens never drawn, the zero-temperature limit equal
  to the masked argmax, and an empty row giving -1.
"""
import math

import numpy as np
import pytest

from oracle import philox4x32_10, ln_f32, mask_sample, mask_logits  # noqa: E402


@pytest.mark.parametrize("ctr,key,out", [
    ((0, 0, 0, 0), (0, 0), (0x6627e8d5, 0xe169c58d, 0xbc57ac4c, 0x9b00dbd8)),
    ((0xffffffff,) * 4, (0xffffffff, 0xffffffff), (0x408f276d, 0x41c83b0e, 0xa20bc7c6, 0x6d5451fd)),
    ((0x243f6a88, 0x85a308d3, 0x13198a2e, 0x03707344), (0xa4093822, 0x299f31d0),
     (0xd16cfe09, 0x94fdcceb, 0x5001e420, 0x24126ea1)),
])
def test_philox_known_answers(ctr, key, out):
    assert tuple(int(x) for x in philox4x32_10(ctr, *key)) == out


def test_ln_f32_accuracy():
    rng = np.random.default_rng(5)
    xs = np.concatenate([np.float32(2.0) ** np.arange(-25, 8).astype(np.float32),
                         rng.uniform(2.0 ** -25, 20.0, 20000).astype(np.float32),
                         (1.0 - np.arange(1, 200) * 2.0 ** -24).astype(np.float32)])
    for x in xs:
        ref = math.log(float(x))
        got = ln_f32(float(x))
        assert abs(got - ref) <= 3e-7 * abs(ref) + 2e-14, (x, got, ref)


def _pack(bits):
    B, V = bits.shape
    W = (V + 31) // 32
    padded = np.zeros((B, W * 32), np.uint8)
    padded[:, :V] = bits
    return np.packbits(padded, axis=1, bitorder="little").view(np.uint32).reshape(B, W)


@pytest.mark.parametrize("temperature", [1.0, 0.5, 2.0])
def test_draws_follow_the_masked_softmax(temperature):
    V, n = 64, 12000
    x = np.zeros((1, V), np.float32)
    allowed = [3, 17, 40, 63]
    x[0, allowed] = [0.0, 1.0, 2.0, 0.5]
    x[0, 5] = 50.0                                     # masked: must never be drawn
    bits = np.zeros((1, V), bool)
    bits[0, allowed] = True
    m = _pack(bits)
    counts = {t: 0 for t in allowed}
    for off in range(n):
        t = int(mask_sample(x, m, temperature, seed=0x1234_5678_9abc, offset=off)[0])
        counts[t] += 1                                 # KeyError if a masked token came out
    p = np.exp(x[0, allowed] / temperature)
    p /= p.sum()
    obs = np.array([counts[t] for t in allowed], float)
    chi2 = float(((obs - n * p) ** 2 / (n * p)).sum())
    assert chi2 < 21.1                                 # 3 degrees of freedom, p = 1e-4


def test_rows_and_seeds_draw_independently():
    V, B = 256, 64
    x = np.zeros((B, V), np.float32)
    m = _pack(np.ones((B, V), bool))
    a = mask_sample(x, m, 1.0, seed=1, offset=0)
    b = mask_sample(x, m, 1.0, seed=2, offset=0)
    c = mask_sample(x, m, 1.0, seed=1, offset=1)
    assert len(set(a.tolist())) > B // 2               # uniform logits: rows differ
    assert len(set((a % 4).tolist())) == 4             # every word of a Philox block is used
    assert (a != b).mean() > 0.9 and (a != c).mean() > 0.9
    assert (a == mask_sample(x, m, 1.0, seed=1, offset=0)).all()


def test_low_temperature_is_the_masked_argmax_and_empty_rows():
    rng = np.random.default_rng(3)
    V, B = 1000, 16
    x = rng.permutation(V * B).reshape(B, V).astype(np.float32)   # distinct, unit-spaced logits
    bits = rng.random((B, V)) < 0.3
    bits[0] = False
    m = _pack(bits)
    arg, _, _ = mask_logits(x, m)
    got = mask_sample(x, m, 1e-3, seed=9, offset=4)
    assert (got == arg).all() and got[0] == -1


def test_bf16_logits_and_row_stride():
    rng = np.random.default_rng(4)
    V, B, stride = 300, 8, 310
    x = rng.standard_normal((B, stride)).astype(np.float32)
    bf = (x.view(np.uint32) >> 16).astype(np.uint16)
    xb = (bf.astype(np.uint32) << 16).view(np.float32)
    m = _pack(rng.random((B, V)) < 0.5)
    a = mask_sample(bf, m, 0.7, seed=11, offset=2, n_tokens=V)
    b = mask_sample(np.ascontiguousarray(xb[:, :V]), m, 0.7, seed=11, offset=2)
    assert (a == b).all()
