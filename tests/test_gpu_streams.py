"""Concurrent use of the library from several CUDA streams.

Several handles (W2, W3, a bit split and a 4-D matrix) run their GEMVs and a
prefill GEMM interleaved on four streams with no synchronisation between the
launches; one handle also runs on two streams at once (the header allows it:
the calls share only the handle's error word).  Every result must equal, bit
for bit, the same call run alone on one stream -- the kernels keep no state
between calls and sum in a fixed order -- and the lone results are checked
against the oracle."""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402


def _dim4_matrix(rows, cols, seed, batch):
    from paper_2609_24875_gb300 import SphqMatrix
    c, x = inp.random_codes_dim(4, 2, rows, cols, seed=seed, B=batch)
    m = SphqMatrix(rows, cols, 2, G.to_dev(c.codebook), G.to_dev(c.scale),
                   G.to_dev(c.offset), radius_bits=c.vbits, K=c.K, dim=4)
    m.pack(G.to_dev(c.sign.astype(np.uint8)), G.to_dev(c.idx), G.to_dev(c.rcode))
    w = oracle.decode_dim(c.codebook, c.scale, c.offset, c.sign, c.idx, c.rcode, c.vbits)
    return m, x, w


def _setup():
    cases = []
    for bits, rv, rows, cols, batch, seed in [(2, None, 1000, 2048, 1, 11),
                                              (3, None, 720, 1024, 4, 12),
                                              (2, (7, 2), 512, 1536, 8, 13)]:
        kw = {}
        if rv is not None:
            kw = dict(radius_bits=rv[1], K=1 << rv[0])
        codes, x = inp.random_codes(bits, rows, cols, seed=seed, B=batch, **kw)
        m = G.make_matrix(codes)
        cases.append((m, x, G.oracle_decode(codes)))
    cases.append(_dim4_matrix(400, 1024, 14, 2))
    return cases


def _lone(m, xd, gemm=False):
    y = m.gemm(xd) if gemm else m.gemv(xd)
    torch.cuda.synchronize()
    return y.clone()


def test_interleaved_streams_match_lone_calls_bit_for_bit():
    cases = _setup()
    xs = [G.x_dev(x) for _, x, _ in cases]
    lone = []
    for (m, x, w), xd in zip(cases, xs):
        y = _lone(m, xd)
        ref, absdot = oracle.gemv(w, x)
        got = y.float().cpu().numpy().astype(np.float64)
        assert np.all(np.abs(got - ref) <= oracle.gemv_tolerance(absdot))
        lone.append(y)
    # a prefill GEMM on the first (8-D W2) matrix alongside the GEMVs
    mg = cases[0][0]
    xg_np = inp.make_x(np.random.default_rng(5), 130, 2048)
    xg = G.x_dev(xg_np)
    yg_lone = _lone(mg, xg, gemm=True)
    ref, absdot = oracle.gemv(cases[0][2], xg_np)
    got = yg_lone.float().cpu().numpy().astype(np.float64)
    assert np.all(np.abs(got - ref) <= oracle.gemv_tolerance(absdot))

    streams = [torch.cuda.Stream() for _ in range(4)]
    reps = 12
    outs = [[torch.empty_like(lone[i]) for _ in range(reps)] for i in range(len(cases))]
    gouts = [torch.empty_like(yg_lone) for _ in range(3)]
    # the W2 handle runs on two streams at once (streams 0 and 3)
    twin = [torch.empty_like(lone[0]) for _ in range(reps)]
    torch.cuda.synchronize()
    for r in range(reps):
        for i, ((m, _, _), xd) in enumerate(zip(cases, xs)):
            m.gemv(xd, y=outs[i][r], stream=streams[i])
        cases[0][0].gemv(xs[0], y=twin[r], stream=streams[3])
        if r % 4 == 0:
            mg.gemm(xg, y=gouts[r // 4], stream=streams[(r // 4) % 4])
    torch.cuda.synchronize()
    for i in range(len(cases)):
        for r in range(reps):
            assert torch.equal(outs[i][r], lone[i]), (i, r)
    for r in range(reps):
        assert torch.equal(twin[r], lone[0]), r
    for y in gouts:
        assert torch.equal(y, yg_lone)
    for m, _, _ in cases:
        m.check()
        m.close()


def test_streams_inside_one_graph():
    """GEMVs of two handles forked onto two streams inside one captured CUDA
    graph (fork/join through events) replay to the lone results."""
    cases = _setup()[:2]
    xs = [G.x_dev(x) for _, x, _ in cases]
    lone = [_lone(m, xd) for (m, _, _), xd in zip(cases, xs)]
    ys = [torch.empty_like(y) for y in lone]
    main = torch.cuda.Stream()
    side = torch.cuda.Stream()
    # warm up outside capture (first calls set kernel attributes)
    with torch.cuda.stream(main):
        cases[0][0].gemv(xs[0], y=ys[0], stream=main)
        cases[1][0].gemv(xs[1], y=ys[1], stream=main)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=main):
        fork = torch.cuda.Event()
        fork.record(main)
        side.wait_event(fork)
        cases[0][0].gemv(xs[0], y=ys[0], stream=main)
        cases[1][0].gemv(xs[1], y=ys[1], stream=side)
        join = torch.cuda.Event()
        join.record(side)
        main.wait_event(join)
    for _ in range(3):
        ys[0].zero_()
        ys[1].zero_()
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(ys[0], lone[0])
        assert torch.equal(ys[1], lone[1])
    for m, _, _ in cases:
        m.check()
        m.close()


def test_sphq_log_reports_formats_and_launch_shapes():
    """SPHQ_LOG=1: creation prints the format and the GEMV plans, a GEMM its
    launch shape (stderr of a child process); unset, nothing is printed."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    prog = (
        "import sys; sys.path[:0] = [%r, %r]\n"
        "import torch, _gpu as G, sphq_inputs as inp\n"
        "c, x = inp.random_codes(3, 64, 512, seed=1, B=1)\n"
        "m = G.make_matrix(c)\n"
        "m.gemm(G.x_dev(inp.make_x(__import__('numpy').random.default_rng(0), 40, 512)))\n"
        "torch.cuda.synchronize(); m.close()\n" % (root, os.path.join(root, "tests")))
    env = dict(os.environ, SPHQ_LOG="1")
    r = subprocess.run([sys.executable, "-c", prog], env=env, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert "sphq: matrix 64 x 512, 8-D, split 8/13/4" in r.stderr
    assert "gemv batch 8:" in r.stderr
    assert "sphq: gemm 64 x 512, batch 40:" in r.stderr
    env["SPHQ_LOG"] = "0"
    r = subprocess.run([sys.executable, "-c", prog], env=env, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert "sphq:" not in r.stderr


@pytest.mark.parametrize("bits,rows,cols,batch", [(2, 1000, 2048, 1), (3, 720, 1024, 2),
                                                  (3, 512, 1536, 8)])
def test_pdl_off_gives_the_same_result(bits, rows, cols, batch):
    """sphq_set_pdl(0): plain stream-ordered launches, same result bit for bit,
    also inside a captured graph of back-to-back GEMVs that feed each other."""
    codes, x = inp.random_codes(bits, rows, cols, seed=4400 + rows + batch, B=batch)
    m = G.make_matrix(codes)
    xd = G.x_dev(x)
    y_on = _lone(m, xd)
    m.set_pdl(False)
    y_off = _lone(m, xd)
    assert torch.equal(y_on, y_off)
    # a chain: each GEMV reads the previous one's output (square matrix)
    sq, _ = inp.random_codes(bits, 256, 256, seed=4500 + batch, B=batch)
    ms = G.make_matrix(sq)
    x0 = G.x_dev(inp.make_x(np.random.default_rng(batch), batch, 256))
    outs = {}
    for pdl in (True, False):
        ms.set_pdl(pdl)
        bufs = [x0.clone()] + [torch.empty_like(x0) for _ in range(4)]
        for i in range(4):
            ms.gemv(bufs[i], y=bufs[i + 1])
        torch.cuda.synchronize()
        outs[pdl] = [b.clone() for b in bufs]
    for a, b in zip(outs[True], outs[False]):
        # bit patterns: late links of the chain may overflow fp16
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    for m_ in (m, ms):
        m_.check()
        m_.close()
