"""Failure detection of the bounded on-chip waits, and export / import of a
packed matrix (neither has a counterpart in the paper).

The wait test makes a wait run out on purpose the way the library allows it:
a kernel waits on an mbarrier nothing arrives on, gives up after about two
seconds, sets the handle's error word and exits; the host reads the status
with sphq_check and the context stays usable (no trap, no fault)."""
import time

import numpy as np
import pytest
import torch

import sphq_inputs as inp
from paper_2609_24875_gb300 import SphqError, SphqMatrix

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402


def test_wait_timeout_is_reported_and_the_context_stays_usable():
    codes, x = inp.random_codes(2, 256, 1024, seed=8, B=2)
    m = G.make_matrix(codes)
    m.check()                                  # clean before
    t0 = time.perf_counter()
    m.selftest_wait_timeout()
    with pytest.raises(SphqError) as e:
        m.check()
    elapsed = time.perf_counter() - t0
    assert e.value.status == 7                 # SPHQ_ERR_TIMEOUT
    assert 1.0 < elapsed < 30.0                # the ~2 s limit, then the kernel returned
    m.check()                                  # the word was cleared by the read
    G.check_gemv(m, codes, x)                  # the context still works
    m.check()
    m.close()


@pytest.mark.parametrize("bits,v,K", [(2, 4, 64), (3, 4, 8192), (3, 3, 8192), (2, 2, 256)])
def test_export_import_round_trip(bits, v, K):
    rows, cols = 300, 1024
    codes, x = inp.random_codes(bits, rows, cols, seed=21 + K + v, B=3, radius_bits=v, K=K)
    m = G.make_matrix(codes)
    blob = m.export()
    m2 = SphqMatrix.from_blob(blob)
    assert (m2.rows, m2.cols, m2.bits, m2.K, m2.radius_bits) == (rows, cols, bits, K, v)
    assert np.array_equal(G.decoded_bits(m2), G.oracle_decode(codes))
    xd = G.x_dev(x)
    y1, y2 = m.gemv(xd).clone(), m2.gemv(xd).clone()
    torch.cuda.synchronize()
    assert torch.equal(y1.view(torch.int16), y2.view(torch.int16))
    assert m2.export() == blob
    m.close()
    m2.close()


def test_import_rejects_malformed_blobs():
    codes, _ = inp.random_codes(2, 32, 256, seed=2)
    m = G.make_matrix(codes)
    blob = m.export()
    for bad in (blob[:40], blob[:-1], b"XXXX" + blob[4:], blob + b"\0"):
        with pytest.raises(SphqError) as e:
            SphqMatrix.from_blob(bad)
        assert e.value.status == 1
    m.close()
