"""GPU parity of alignment/correction (Eq. 4-7) and gated fusion (Eq. 8) vs the oracle.

Covers both kernel families: the tcgen05 tensor-core path (bf16, d a multiple
of 256) and the FFMA path (fp32, and bf16 at other hidden sizes).
"""

import math

import numpy as np
import pytest
import torch

import oracle
from parity import assert_close, host_f64, host_int

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rt():
    from paper_2608_29748_gb300 import binding

    return binding


def make_inputs(B, K, d, dtype, seed, accept=None):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    hD = torch.randn((B, K, d), generator=g, device="cuda").to(dtype)
    hT = torch.randn((B, K, d), generator=g, device="cuda").to(dtype)
    a = math.sqrt(2.0 / d)
    Wc = ((torch.rand((d, 2 * d), generator=g, device="cuda") * 2 - 1) * a).to(dtype)
    Wv = ((torch.rand((d, d), generator=g, device="cuda") * 2 - 1) * math.sqrt(3.0 / d)).to(dtype)
    Wg = ((torch.rand((d, 2 * d), generator=g, device="cuda") * 2 - 1) * a).to(dtype)
    e_vec = (torch.randn((d,), generator=g, device="cuda") * 0.02).to(dtype)
    e_dense = (torch.randn((B, K, d), generator=g, device="cuda") * 0.02).to(dtype)
    if accept is None:
        edge = torch.tensor([0, K - 2, K - 1, K], device="cuda").clamp(min=0)
        accept = torch.randint(0, K + 1, (B,), generator=g, device="cuda")
        accept[: min(B, 4)] = edge[: min(B, 4)]
    return dict(hD=hD, hT=hT, Wc=Wc, Wv=Wv, Wg=Wg, e_vec=e_vec, e_dense=e_dense,
                accept=accept.to(torch.int32))


SHAPES = [
    # (B, K, d, dtype)  -- tensor-core path
    (1, 16, 256, torch.bfloat16),
    (5, 4, 512, torch.bfloat16),
    (19, 16, 256, torch.bfloat16),  # 19 * 15 = 285 rows: 3 M tiles, ragged last tile
    (3, 16, 2560, torch.bfloat16),
    # FFMA path
    (4, 8, 192, torch.bfloat16),
    (3, 5, 100, torch.bfloat16),
    (2, 8, 256, torch.float32),
    (6, 16, 96, torch.float32),
    (4, 9, 160, torch.float32),  # B (K-1) = 32: the last shape of the warp-per-feature kernel
    (3, 12, 160, torch.bfloat16),  # B (K-1) = 33: the first of the 32 x 64 tiles
]


@pytest.mark.parametrize("B,K,d,dtype", SHAPES)
def test_align_refine(rt, B, K, d, dtype):
    x = make_inputs(B, K, d, dtype, seed=B * 7 + K + d)
    beta = 0.75
    r = torch.full((B, K, d), 9.0, dtype=dtype, device="cuda")
    n = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    ws = rt.Workspace(B, K, 8, d, dtype)
    rt.retrace_align_refine(x["hD"], x["hT"], x["accept"], x["Wc"], beta, r, n, ws)
    torch.cuda.synchronize()
    assert ws.check() == 0
    A = host_int(x["accept"])
    np.testing.assert_array_equal(host_int(n), oracle.carried_rows(A, K))
    m, u = oracle.align(host_f64(x["hD"]), host_f64(x["hT"]), A)
    want = oracle.correct(m, u, host_f64(x["Wc"]), beta, round_r_bf16=False)
    assert_close(r, want, "r")
    # rows that carry nothing are exactly zero (Eq. 4-5 zero padding)
    got = host_f64(r)
    for b in range(B):
        assert not got[b, oracle.carried_rows(A, K)[b]:].any()


def test_align_refine_clamps_out_of_range_accept(rt):
    B, K, d = 4, 6, 256
    acc = torch.tensor([-3, 0, K + 5, 2], dtype=torch.int32, device="cuda")
    x = make_inputs(B, K, d, torch.bfloat16, seed=5, accept=acc)
    r = torch.empty((B, K, d), dtype=torch.bfloat16, device="cuda")
    n = torch.empty((B,), dtype=torch.int32, device="cuda")
    ws = rt.Workspace(B, K, 8, d, torch.bfloat16)
    rt.retrace_align_refine(x["hD"], x["hT"], acc, x["Wc"], 1.0, r, n, ws)
    torch.cuda.synchronize()
    clamped = np.clip(host_int(acc), 0, K)
    np.testing.assert_array_equal(host_int(n), oracle.carried_rows(clamped, K))
    m, u = oracle.align(host_f64(x["hD"]), host_f64(x["hT"]), clamped)
    assert_close(r, oracle.correct(m, u, host_f64(x["Wc"]), 1.0, False), "r")


@pytest.mark.parametrize("dense_e", [False, True])
@pytest.mark.parametrize("B,K,d,dtype", SHAPES)
def test_gate_fuse(rt, B, K, d, dtype, dense_e):
    x = make_inputs(B, K, d, dtype, seed=B + K * 3 + d + int(dense_e))
    g = torch.Generator(device="cuda")
    g.manual_seed(d)
    r = torch.randn((B, K, d), generator=g, device="cuda").to(dtype)
    n = torch.from_numpy(oracle.carried_rows(host_int(x["accept"]), K).astype(np.int32)).cuda()
    e = x["e_dense"] if dense_e else x["e_vec"]
    out = torch.full((B, K, d), 7.0, dtype=dtype, device="cuda")
    ws = rt.Workspace(B, K, 8, d, dtype)
    rt.retrace_gate_fuse(e, r, n, x["Wv"], x["Wg"], out, ws)
    torch.cuda.synchronize()
    assert ws.check() == 0
    e_full = np.broadcast_to(host_f64(e), (B, K, d))
    want = oracle.gate_fuse(e_full, host_f64(r), host_int(n), host_f64(x["Wv"]), host_f64(x["Wg"]))
    assert_close(out, want, "e_tilde")
    got = host_f64(out)
    for b in range(B):
        nb = int(n[b])
        assert np.array_equal(got[b, nb:], e_full[b, nb:])  # unconditioned rows keep e exactly


@pytest.mark.parametrize("d,dtype", [(256, torch.bfloat16), (512, torch.bfloat16), (192, torch.bfloat16), (256, torch.float32)])
def test_closed_gate_reproduces_e_exactly(rt, d, dtype):
    """W_v = 0 (the paper's initialisation): e~ == e bit-for-bit on every row."""
    B, K = 7, 16
    x = make_inputs(B, K, d, dtype, seed=3)
    r = torch.randn((B, K, d), device="cuda").to(dtype)
    n = torch.full((B,), K - 1, dtype=torch.int32, device="cuda")
    out = torch.empty((B, K, d), dtype=dtype, device="cuda")
    ws = rt.Workspace(B, K, 8, d, dtype)
    rt.retrace_gate_fuse(x["e_vec"], r, n, torch.zeros_like(x["Wv"]), x["Wg"], out, ws)
    torch.cuda.synchronize()
    assert torch.equal(out, x["e_vec"].expand(B, K, d))


@pytest.mark.parametrize("d,dtype", [(256, torch.bfloat16), (192, torch.bfloat16), (256, torch.float32)])
def test_half_gate_identity_value_is_exact(rt, d, dtype):
    """W_g = 0, W_v = I, beta = 0: e~ = e + m/2 (Eq. 7-8 closed form), rows without signal keep e."""
    B, K = 5, 8
    x = make_inputs(B, K, d, dtype, seed=11)
    eye = torch.eye(d, device="cuda").to(dtype)
    r = torch.empty((B, K, d), dtype=dtype, device="cuda")
    n = torch.empty((B,), dtype=torch.int32, device="cuda")
    out = torch.empty((B, K, d), dtype=dtype, device="cuda")
    ws = rt.Workspace(B, K, 8, d, dtype)
    rt.retrace_align_refine(x["hD"], x["hT"], x["accept"], x["Wc"], 0.0, r, n, ws)
    rt.retrace_gate_fuse(x["e_vec"], r, n, eye, torch.zeros_like(x["Wg"]), out, ws)
    torch.cuda.synchronize()
    A = host_int(x["accept"])
    m, _ = oracle.align(host_f64(x["hD"]), host_f64(x["hT"]), A)
    e_full = np.broadcast_to(host_f64(x["e_vec"]), (B, K, d))
    # v = r = m and sigmoid(0) = 1/2 are exact on both sides; the only rounding
    # left is the fp32 addition (then bf16 for bf16 outputs), mirrored here.
    want = (e_full.astype(np.float32) + (0.5 * m).astype(np.float32)).astype(np.float64)
    got = host_f64(out)
    if dtype == torch.bfloat16:
        want = oracle.round_to_bf16(want)
    assert np.array_equal(got, want)


def accept_for_rows(B, K, R):
    """Accepted lengths whose carried rows n_b = max(0, K-1-A_b) sum to R."""
    a = torch.full((B,), K, dtype=torch.int32)
    left = R
    for b in range(B):
        n = min(K - 1, left)
        a[b] = K - 1 - n if n > 0 else K
        left -= n
    assert left == 0
    return a.cuda()


@pytest.mark.parametrize("R", [1, 15, 16, 17, 127, 128, 129, 240, 241, 255, 256, 257, 384, 513, 769, 1023, 1200])
def test_pair_tile_boundaries(rt, R):
    """Row counts around the tile edges of the CTA-pair kernel: one to five
    row tiles of 16 to 256 rows (a multiple of 16 chosen from R), halves of
    8 to 128 rows in each CTA loaded as boxes of 64, 32, 16 and 8 rows, and
    the last tile's padding.  B (K-1) = 1200 possible rows keeps the call off
    the small-R path."""
    B, K, d, dtype = 80, 16, 256, torch.bfloat16
    x = make_inputs(B, K, d, dtype, seed=R, accept=accept_for_rows(B, K, R))
    A = host_int(x["accept"])
    n_host = oracle.carried_rows(A, K)
    assert n_host.sum() == R
    ws = rt.Workspace(B, K, 8, d, dtype)
    r = torch.full((B, K, d), 9.0, dtype=dtype, device="cuda")
    n = torch.empty((B,), dtype=torch.int32, device="cuda")
    rt.retrace_align_refine(x["hD"], x["hT"], x["accept"], x["Wc"], 0.5, r, n, ws)
    out = torch.full((B, K, d), 7.0, dtype=dtype, device="cuda")
    rt.retrace_gate_fuse(x["e_vec"], r, n, x["Wv"], x["Wg"], out, ws)
    torch.cuda.synchronize()
    assert ws.check() == 0
    m, u = oracle.align(host_f64(x["hD"]), host_f64(x["hT"]), A)
    r_ref = oracle.correct(m, u, host_f64(x["Wc"]), 0.5, round_r_bf16=False)
    assert_close(r, r_ref, f"r, R={R}")
    e_full = np.broadcast_to(host_f64(x["e_vec"]), (B, K, d))
    want = oracle.gate_fuse(e_full, host_f64(r), n_host, host_f64(x["Wv"]), host_f64(x["Wg"]))
    assert_close(out, want, f"e~, R={R}")


@pytest.mark.parametrize("B,K,d", [(1, 2, 256), (3, 6, 512), (16, 16, 256), (16, 17, 256), (8, 16, 2560),
                                   (17, 16, 256), (40, 16, 256), (64, 17, 256)])
def test_small_r_path(rt, B, K, d):
    """At most 1024 conditioned rows (B (K-1) <= 1024): the GEMMs run with the
    weights as the 128-row side against N tiles of up to 256 rows, split over
    K, the partials summed in a fixed order.  Every draft rejected at once
    (A_b = 0), so all B (K-1) rows are carried: 1, 15, 240, 256, 255, 600 and
    1024 rows (one to four N tiles, the last one partial) and d up to 2560;
    both entry points against the oracle, repeatable bit for bit."""
    dtype = torch.bfloat16
    x = make_inputs(B, K, d, dtype, seed=B * 100 + K, accept=torch.zeros(B, dtype=torch.int32).cuda())
    A = host_int(x["accept"])
    n_host = oracle.carried_rows(A, K)
    assert n_host.sum() == B * (K - 1)
    ws = rt.Workspace(B, K, 8, d, dtype)
    outs = []
    for _ in range(2):
        r = torch.full((B, K, d), 9.0, dtype=dtype, device="cuda")
        n = torch.empty((B,), dtype=torch.int32, device="cuda")
        rt.retrace_align_refine(x["hD"], x["hT"], x["accept"], x["Wc"], 0.75, r, n, ws)
        out = torch.full((B, K, d), 7.0, dtype=dtype, device="cuda")
        rt.retrace_gate_fuse(x["e_vec"], r, n, x["Wv"], x["Wg"], out, ws)
        torch.cuda.synchronize()
        outs.append((r, out))
    assert ws.check() == 0
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])
    r, out = outs[0]
    m, u = oracle.align(host_f64(x["hD"]), host_f64(x["hT"]), A)
    r_ref = oracle.correct(m, u, host_f64(x["Wc"]), 0.75, round_r_bf16=False)
    assert_close(r, r_ref, f"r, B={B} K={K}")
    e_full = np.broadcast_to(host_f64(x["e_vec"]), (B, K, d))
    want = oracle.gate_fuse(e_full, host_f64(r), n_host, host_f64(x["Wv"]), host_f64(x["Wg"]))
    assert_close(out, want, f"e~, B={B} K={K}")


@pytest.mark.parametrize("B,K,d,R", [(1, 2, 256, 1), (1, 17, 512, 15), (2, 9, 256, 16), (17, 2, 1024, 17),
                                     (8, 16, 4096, 100), (16, 16, 256, 240), (17, 16, 2560, 255),
                                     (16, 17, 256, 256),
                                     # more than 256 possible rows: N tiles of 256, split-K partials
                                     (18, 16, 256, 16), (18, 16, 512, 257), (40, 16, 256, 511),
                                     (40, 16, 1024, 512), (35, 16, 4096, 513), (64, 16, 2560, 960),
                                     (64, 17, 256, 1000), (64, 17, 512, 1024)])
def test_small_r_rows(rt, B, K, d, R):
    """Exactly R carried rows on the small-R path (B (K-1) <= 1024).  At most
    256 possible rows the GEMMs run as split-K clusters that sum their
    partials through distributed shared memory; above that as split-K tiles
    whose fp32 partials a reduction kernel sums.  R below, at and above
    multiples of 16 and of 256 (one to four N tiles), cluster sizes that
    differ between d = 256 and d = 4096: r and e~ against the oracle through
    both standalone entry points, and repeated bit for bit."""
    dtype = torch.bfloat16
    assert B * (K - 1) <= 1024 and R <= B * (K - 1)
    # carry exactly R rows: sequences reject at once (n_b = K - 1) until R is reached
    n_want = np.zeros(B, dtype=np.int64)
    left = R
    for b in range(B):
        n_want[b] = min(K - 1, left)
        left -= n_want[b]
    accept = torch.tensor([K - 1 - n if n > 0 else K for n in n_want], dtype=torch.int32).cuda()
    x = make_inputs(B, K, d, dtype, seed=1000 + R + d, accept=accept)
    A = host_int(x["accept"])
    n_host = oracle.carried_rows(A, K)
    assert int(n_host.sum()) == R
    ws = rt.Workspace(B, K, 8, d, dtype)
    outs = []
    for _ in range(2):
        r = torch.full((B, K, d), 9.0, dtype=dtype, device="cuda")
        n = torch.empty((B,), dtype=torch.int32, device="cuda")
        rt.retrace_align_refine(x["hD"], x["hT"], x["accept"], x["Wc"], 0.5, r, n, ws)
        out = torch.full((B, K, d), 7.0, dtype=dtype, device="cuda")
        rt.retrace_gate_fuse(x["e_vec"], r, n, x["Wv"], x["Wg"], out, ws)
        torch.cuda.synchronize()
        outs.append((r, out))
    assert ws.check() == 0
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])
    r, out = outs[0]
    m, u = oracle.align(host_f64(x["hD"]), host_f64(x["hT"]), A)
    r_ref = oracle.correct(m, u, host_f64(x["Wc"]), 0.5, round_r_bf16=False)
    assert_close(r, r_ref, f"r, R={R} d={d}")
    e_full = np.broadcast_to(host_f64(x["e_vec"]), (B, K, d))
    want = oracle.gate_fuse(e_full, host_f64(r), n_host, host_f64(x["Wv"]), host_f64(x["Wg"]))
    assert_close(out, want, f"e~, R={R} d={d}")
