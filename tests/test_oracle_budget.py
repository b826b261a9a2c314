"""Pins of the bit-budget formulas against the numbers the paper prints
(§3.1, §3.2, Tab. 4, Tab. 7, App. B / Tab. 12) in tests/golden/bit_budget.txt."""
import os

import pytest

import oracle
import sphq_inputs as inp

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rows():
    with open(os.path.join(GOLDEN, "bit_budget.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            p = line.split()
            kw = dict(t.split("=") for t in p[1:-1])
            yield p[0], {k: int(v) for k, v in kw.items()}, float(p[-1])


@pytest.mark.parametrize("kind,kw,expected", list(_rows()))
def test_budget(kind, kw, expected):
    if kind == "entries":
        assert oracle.codebook_entries(kw["bits"], kw["dim"]) == expected
    elif kind == "cbbytes":
        assert oracle.codebook_bytes(kw["bits"], kw["dim"], bool(kw["signed"])) == expected
    elif kind == "payload":
        assert oracle.payload_bits_per_weight(kw["bits"], kw["V"]) == expected
    elif kind == "split":
        assert (kw["sign"] + kw["dir"] + kw["radius"]) / 8 == expected
        assert oracle.split_bits_per_weight(kw["dir"], kw["radius"]) == expected
        # §3.2: the same budget is 2 + (V - 2)/8 when the index keeps 6 bits
        if kw["dir"] == 6:
            assert 2 + (kw["radius"] - 2) / 8 == expected
    else:  # pragma: no cover
        raise AssertionError(kind)


def test_generator_codebook_sizes_follow_the_budget():
    for bits in (2, 3):
        assert inp.bits_to_K(bits) == oracle.codebook_entries(bits)
