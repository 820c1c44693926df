"""Pins of the oracle's 4-bit compression (Section 3, 'Base model weights compression').

The oracle is checked against a hand-worked example, the round-trip error
bound, idempotence on its own decode, range facts and (for the fp16 operand
value) torch's own round-to-nearest-even conversion.
"""
import json
import os

import numpy as np
import pytest

from oracle import quant

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _worked():
    with open(os.path.join(GOLD, "quant_worked_example.json")) as f:
        g = json.load(f)
    W = np.zeros((g["rows"], g["cols"]), np.float32)
    for e in g["nonzero"]:
        W[e["row"], e["col"]] = e["w"]
    return g, W


def test_hand_worked_example():
    g, W = _worked()
    qpack, scales = quant.compress(W)
    assert qpack.shape == (2, 64) and scales.shape == (2, 2)
    assert scales.view(np.uint16).tolist() == g["scales_fp16_bits_group_major"]
    assert qpack[0, :4].tolist() == g["qpack_row0_head"]
    assert qpack[1, :4].tolist() == g["qpack_row1_head"]
    assert qpack[1, 32:36].tolist() == g["qpack_row1_group1_head"]
    q = quant.unpack_codes(qpack)
    expect = np.zeros_like(q)
    for e in g["codes_nonzero"]:
        expect[e["row"], e["col"]] = e["q"]
    np.testing.assert_array_equal(q, expect)
    # every untouched byte is the zero code (u = 8 in both nibbles)
    assert (qpack[0, 4:] == 0x88).all()


def test_word_layout_is_even_columns_low_half_odd_columns_high_half():
    """Element 8w+2j sits in bits 4j..4j+3 of little-endian word w, element 8w+2j+1 in bits 16+4j.."""
    W = np.zeros((1, 64), np.float32)
    W[0, :8] = [-7, -5, -3, -1, 1, 3, 5, 7]
    W[0, 8] = 7.0
    qpack, scales = quant.compress(W)
    assert float(scales[0, 0]) == 1.0
    word = int(qpack[0, :4].view("<u4")[0])
    u = [(word >> (4 * j)) & 0xF for j in range(4)] + [(word >> (16 + 4 * j)) & 0xF for j in range(4)]
    assert u == [1, 5, 9, 13, 3, 7, 11, 15]          # even columns 0,2,4,6 then odd 1,3,5,7
    np.testing.assert_array_equal(quant.unpack_codes(qpack)[0, :8], [-7, -5, -3, -1, 1, 3, 5, 7])


def _rand(rows, cols, seed, std=0.02):
    return (np.random.default_rng(seed).standard_normal((rows, cols)) * std).astype(np.float32)


@pytest.mark.parametrize("seed", [0, 1])
def test_round_trip_bound(seed):
    W = _rand(64, 512, seed)
    W[3, 64:128] *= 1e3        # a loud group
    W[5, :64] = 0.0            # an all-zero group
    qpack, scales = quant.compress(W)
    deq = quant.dequant(qpack, scales)
    s = quant.row_scales(scales).astype(np.float64)
    err = np.abs(deq - W.astype(np.float64))
    assert (err <= 0.5 * s * (1 + 1e-6) + 1e-30).all()
    assert (deq[5, :64] == 0).all()


def test_codes_in_symmetric_range_and_nibbles_nonzero():
    W = _rand(32, 256, 7, std=1.0)
    qpack, _ = quant.compress(W)
    q = quant.unpack_codes(qpack)
    assert q.min() >= -7 and q.max() <= 7
    assert ((qpack & 0x0F) != 0).all() and ((qpack >> 4) != 0).all()
    # each group holds a +-7 (the element with the largest magnitude)
    assert (np.abs(q.reshape(32, -1, 64)).max(axis=2) == 7).all()


def test_idempotent_on_its_own_decode():
    W = _rand(48, 320, 3)
    qpack, scales = quant.compress(W)
    deq32 = quant.dequant(qpack, scales).astype(np.float32)   # q*s is exact in fp32
    qpack2, scales2 = quant.compress(deq32)
    np.testing.assert_array_equal(qpack, qpack2)
    np.testing.assert_array_equal(scales.view(np.uint16), scales2.view(np.uint16))


def test_scale_saturates_to_fp16_max():
    W = np.zeros((1, 64), np.float32)
    W[0, 0] = 1e6
    qpack, scales = quant.compress(W)
    assert float(scales[0, 0]) == 65504.0
    assert quant.unpack_codes(qpack)[0, 0] == 7     # clamped code


def test_f16_operand_bits_match_torch_rne():
    torch = pytest.importorskip("torch")
    W = _rand(16, 256, 11, std=0.5)
    W[0, :64] *= 1e-6          # scales in the fp16 subnormal range
    qpack, scales = quant.compress(W)
    bits = quant.dequant_f16_bits(qpack, scales)
    deq32 = torch.from_numpy(quant.dequant(qpack, scales).astype(np.float32))
    tb = deq32.to(torch.float16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(bits, tb)
    np.testing.assert_array_equal(quant.f16_bits_to_f64(bits), tb.view(np.float16).astype(np.float64))


def test_rejects_ragged_groups():
    with pytest.raises(ValueError):
        quant.compress(np.zeros((2, 96), np.float32))
