"""Pins of the paper's W2 word format (§3.4, Fig. 3(b)): hand-derived words
from tests/golden/w2_words.txt and a pack/unpack round trip."""
import os

import numpy as np

import oracle
import sphq_inputs as inp

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_w2_word_fixture():
    sign = np.zeros((1, 16), np.uint8)
    idx = np.zeros((1, 16), np.uint16)
    rcode = np.zeros((1, 16), np.uint8)
    expect_base = np.zeros(16, np.uint16)
    expect_extra = None
    with open(os.path.join(GOLDEN, "w2_words.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            p = line.split()
            if p[0] == "EXTRA":
                expect_extra = int(p[1], 16)
                continue
            j = int(p[0])
            sign[0, j], idx[0, j], rcode[0, j] = int(p[1], 16), int(p[2]), int(p[3])
            expect_base[j] = int(p[4], 16)
    base, extra = oracle.pack_w2_words(sign, idx, rcode)
    assert np.array_equal(base[0], expect_base)
    assert int(extra[0, 0]) == expect_extra


def test_w2_words_round_trip_and_size():
    codes, _ = inp.random_codes(2, 6, 512, seed=31)
    base, extra = oracle.pack_w2_words(codes.sign, codes.idx, codes.rcode)
    s, i, r = oracle.unpack_w2_words(base, extra)
    assert np.array_equal(s, codes.sign)
    assert np.array_equal(i, codes.idx)
    assert np.array_equal(r, codes.rcode)
    # 16 bits per vector + 32 bits per 16 vectors = 2.25 bits per weight (App. B)
    bits = base.nbytes * 8 + extra.nbytes * 8
    assert bits / (6 * 512) == 2.25 == oracle.payload_bits_per_weight(2, 4)
