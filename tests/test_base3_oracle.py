"""CPU pins of the oracle's base-3 storage of ternary codes (5 trits per
byte; eq. (14)'s ~1.58-bit accounting): hand-computed bytes, the bijection
between the 243 byte values and the 5-trit words, the storage rate against
eq. (14), padding, round trips and the invalid-byte count."""
import itertools

import numpy as np
import pytest

import oracle as O


def test_hand_computed_bytes():
    # trits 1, 2, 0, 0, 1 -> 1 + 2*3 + 0*9 + 0*27 + 1*81 = 88
    codes = np.array([[1, -1, 0, 0, 1]], dtype=np.int8)
    assert O.pack_base3(codes)[0, 0] == 88
    # all -1: 2 * (1 + 3 + 9 + 27 + 81) = 242, the largest valid byte
    assert O.pack_base3(-np.ones((1, 5), dtype=np.int8))[0, 0] == 242
    # code j = 7 sits at digit 2 of byte 1
    c = np.zeros((1, 10), dtype=np.int8)
    c[0, 7] = 1
    b = O.pack_base3(c)
    assert b[0, 0] == 0 and b[0, 1] == 9


def test_all_243_words_round_trip_uniquely():
    words = np.array(list(itertools.product([0, 1, -1], repeat=5)), dtype=np.int8)
    b = O.pack_base3(words)[:, 0]
    assert sorted(b.tolist()) == list(range(243))
    back, bad = O.unpack_base3(O.pack_base3(words), 5)
    assert bad == 0 and np.array_equal(back, words)


def test_storage_rate_against_eq14():
    # 8 bits / 5 trits = 1.6 bits per code, above log2(3) = 1.585 (eq. (14)'s 1.58)
    assert 8 / O.TRITS_PER_BYTE == 1.6
    assert 3 ** O.TRITS_PER_BYTE <= 256 < 3 ** 6
    assert abs(O.compression_ratio(1.6, 2.0) - 0.2) < 1e-12
    k = 16384
    assert O.base3_bytes_per_row(k) * 8 / k <= 1.6 + 16 * 8 / k
    assert O.base3_bytes_per_row(k) < O.plain_words_per_row(k, O.TERNARY) * 4 * 0.81


@pytest.mark.parametrize("k", [1, 5, 79, 80, 81, 256, 320, 1000])
def test_round_trip_and_padding(k):
    rng = np.random.default_rng(k)
    c = rng.integers(-1, 2, size=(7, k)).astype(np.int8)
    b = O.pack_base3(c)
    assert b.shape == (7, O.base3_bytes_per_row(k)) and b.shape[1] % 16 == 0
    assert b.max() <= 242
    # bytes past the last code are 0, and so are the trits past K_eff
    nb = -(-k // 5)
    assert np.all(b[:, nb:] == 0)
    if k % 5:
        assert np.all(b[:, nb - 1] < 3 ** (k % 5))
    back, bad = O.unpack_base3(b, k)
    assert bad == 0 and np.array_equal(back, c)


def test_invalid_bytes_counted_and_read_as_zero():
    b = np.zeros((2, 16), dtype=np.uint8)
    b[0, 0] = 243
    b[1, 3] = 255
    b[1, 4] = 88
    codes, bad = O.unpack_base3(b, 25)
    assert bad == 2
    assert np.all(codes[0, :5] == 0) and np.all(codes[1, 15:20] == 0)
    assert codes[1, 20:25].tolist() == [1, -1, 0, 0, 1]
