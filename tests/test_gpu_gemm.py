"""GPU parity: the tcgen05 GEMM candidate (and the SIMT reference) against the
oracle's fp64 GEMM: exact on identity / permutation / small-integer inputs,
within |d| <= 2^-7 |ref| + 2^-12 sqrt(K) element by element on seeded inputs
(ragged tails, several tiles and waves), on seeded samples at the large sizes."""
import math

import numpy as np
import pytest
import torch

import paper_2609_30057_gb300 as krex
from gpu_util import Guarded, bits16, to_bf16_tensor, to_f16_tensor
import inputs
from oracle import gen, ref

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    krex.build()


@pytest.fixture(autouse=True)
def default_tuning():
    """Every test starts and ends with the library's default tuning."""
    krex.krex_set_tuning()
    yield
    krex.krex_set_tuning()


@pytest.fixture(params=["2", "2k1"], ids=["2sm", "2sm_ksub1"])
def variant(request):
    """The tcgen05 kernel's two stage depths: 128-deep stages (default) and
    64-deep stages."""
    krex.krex_set_tuning(gemm_stage_k=64 if request.param == "2k1" else 128)
    return request.param


def _gen(seed, M, N, K):
    a = torch.empty(M, K, dtype=torch.bfloat16, device="cuda")
    b = torch.empty(K, N, dtype=torch.bfloat16, device="cuda")
    krex.krex_gen_inputs(seed, 0, krex.KREX_DIST_UNIFORM_PM1, 0.0, a)
    krex.krex_gen_inputs(seed, 1, krex.KREX_DIST_UNIFORM_PM1, 0.0, b)
    return a, b


def _candidate(a, b, guard=True):
    M, N = a.shape[0], b.shape[1]
    c = Guarded(M, N, torch.bfloat16) if guard else None
    out = c.view if guard else torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    krex.krex_run_candidate(krex.KREX_OP_GEMM_BF16, [a, b], out)
    torch.cuda.synchronize()
    assert krex.krex_device_status() == 0
    if guard:
        assert c.canaries_intact()
    return out


def _within_tol(got_bits, want64, K):
    got = gen.bf16_to_f32(got_bits).astype(np.float64)
    err = np.abs(got - want64)
    tol = ref.gemm_tolerance(want64, K)
    return np.all(err <= tol), float(np.max(err / tol))


def test_identity_is_exact(variant):
    n = 256
    a, _ = _gen(1, 256, n, 384)
    eye = to_bf16_tensor(inputs.bf16_bits_from_f32(inputs.identity(384)))
    c = _candidate(a, eye)
    assert np.array_equal(bits16(c), bits16(a))


def test_permutation_is_exact(variant):
    a, _ = _gen(2, 128, 512, 512)
    p, perm = inputs.permutation_matrix(512, 9)
    c = _candidate(a, to_bf16_tensor(inputs.bf16_bits_from_f32(p)))
    assert np.array_equal(bits16(c), bits16(a)[:, perm])


def test_small_integers_are_exact(variant):
    # integer operands in [-4, 4]: every partial sum is an integer < 2^8 * K,
    # exact in fp32; outputs below 256 are exact in bf16
    M, N, K = 256, 512, 64
    g = inputs.rng(4)
    a = g.integers(-4, 5, (M, K)).astype(np.float32)
    b = g.integers(-4, 5, (K, N)).astype(np.float32)
    ab, bb = inputs.bf16_bits_from_f32(a), inputs.bf16_bits_from_f32(b)
    c = _candidate(to_bf16_tensor(ab), to_bf16_tensor(bb))
    want = ref.gemm_f64(ab, bb)
    assert np.max(np.abs(want)) < 256
    assert np.array_equal(gen.bf16_to_f32(bits16(c)).astype(np.float64), want)


@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (128, 256, 128), (256, 512, 256), (100, 72, 40), (512, 512, 192),
                                   (129, 264, 136), (1, 8, 8), (300, 1000, 520), (1024, 2048, 512),
                                   (2048, 4096, 1024), (640, 384, 4104)])
def test_seeded_gemm_within_tolerance(M, N, K, variant):
    seed = 1000 + M + N + K
    a, b = _gen(seed, M, N, K)
    c = _candidate(a, b)
    want = ref.gemm_f64(gen.uniform_bf16(seed, 0, M, K), gen.uniform_bf16(seed, 1, K, N))
    ok, worst = _within_tol(bits16(c), want, K)
    assert ok, worst


@pytest.mark.parametrize("bn", [128, 192, 256, 512])
@pytest.mark.parametrize("M,N,K", [(300, 1000, 520), (512, 1792, 256), (256, 192, 64), (260, 328, 72)])
def test_2sm_every_pair_tile_width(M, N, K, bn):
    krex.krex_set_tuning(gemm_pair_tile_n=bn)
    seed = 3000 + M + N + K
    a, b = _gen(seed, M, N, K)
    c = _candidate(a, b)
    want = ref.gemm_f64(gen.uniform_bf16(seed, 0, M, K), gen.uniform_bf16(seed, 1, K, N))
    ok, worst = _within_tol(bits16(c), want, K)
    assert ok, worst


@pytest.mark.parametrize("M,N,K", [(2048, 4096, 4096), (1000, 3000 - 8, 1032), (4096, 4096, 4096)])
def test_wide_pair_tiles_several_waves(M, N, K):
    # pair tiles of 256 x 512 (two MMAs of N = 256 per K step into one
    # 512-column accumulator, the epilogue draining it before the next tile):
    # several tiles per pair, a ragged last column chunk, full output; and the
    # same GEMM through the workspace form, both K orders
    krex.krex_set_tuning(gemm_pair_tile_n=512)
    seed = 3500 + M + N + K
    a, b = _gen(seed, M, N, K)
    want = ref.gemm_f64(gen.uniform_bf16(seed, 0, M, K), gen.uniform_bf16(seed, 1, K, N))
    c = _candidate(a, b)
    ok, worst = _within_tol(bits16(c), want, K)
    assert ok, worst
    for alt in (0, 1):
        krex.krex_set_tuning(gemm_pair_tile_n=512, gemm_k_alternate=alt)
        g = Guarded(M, N, torch.bfloat16)
        krex.krex_run_candidate_ws(krex.KREX_OP_GEMM_BF16, [a, b], g.view, krex.gemm_workspace())
        torch.cuda.synchronize()
        assert krex.krex_device_status() == 0 and g.canaries_intact()
        ok, worst = _within_tol(bits16(g.view), want, K)
        assert ok, worst


def test_wide_pair_tiles_f16_and_large_sampled():
    krex.krex_set_tuning(gemm_pair_tile_n=512)
    M, N, K = 1536, 2560, 2048
    ah, bh = gen.uniform_f16(71, 0, M, K), gen.uniform_f16(71, 1, K, N)
    c = Guarded(M, N, torch.float16)
    krex.krex_run_candidate(krex.KREX_OP_GEMM_F16, [to_f16_tensor(ah), to_f16_tensor(bh)], c.view)
    torch.cuda.synchronize()
    assert krex.krex_device_status() == 0 and c.canaries_intact()
    want = ref.gemm_f64(ah, bh, dtype="f16")
    got = gen.f16_to_f32(bits16(c.view)).astype(np.float64)
    assert np.all(np.abs(got - want) <= ref.gemm_tolerance(want, K, dtype="f16"))
    n = 16384
    a, b = _gen(5, n, n, n)
    out = _candidate(a, b, guard=False)
    i, j = ref.sample_indices(5, 2, 4096, n, n)
    got = bits16(out[torch.from_numpy(i).cuda(), torch.from_numpy(j).cuda()])
    ok, worst = _within_tol(got, ref.gemm_sampled_f64(5, n, n, n, i, j), n)
    assert ok, worst


@pytest.mark.parametrize("ldc_pad", [0, 8, 4, 3])
def test_output_row_stride(ldc_pad, variant):
    # ldc a multiple of 8: TMA-store epilogue; otherwise direct stores.  The
    # sentinel bands (and the padding columns between rows) must stay intact.
    M, N, K = 300, 520, 136
    seed = 4000 + ldc_pad
    a, b = _gen(seed, M, N, K)
    c = Guarded(M, N, torch.bfloat16, ld=N + ldc_pad)
    krex.krex_run_candidate(krex.KREX_OP_GEMM_BF16, [a, b], c.view)
    torch.cuda.synchronize()
    assert krex.krex_device_status() == 0
    assert c.canaries_intact()
    want = ref.gemm_f64(gen.uniform_bf16(seed, 0, M, K), gen.uniform_bf16(seed, 1, K, N))
    ok, worst = _within_tol(bits16(c.view), want, K)
    assert ok, worst


@pytest.mark.parametrize("tun", [{}, {"gemm_pair_tile_n": 512}, {"gemm_pair_tile_n": 256, "gemm_stage_k": 64},
                                 {"gemm_pair_tile_n": 192}], ids=["auto", "wide", "k64", "n192"])
def test_seeded_random_shapes(tun):
    # twelve shapes drawn from a seeded generator (M, N, K multiples of 8 up
    # to 2.5k, some tiny), each within tolerance of the oracle, through the
    # workspace form (K halves where they apply)
    rng = np.random.default_rng(20261202)
    krex.krex_set_tuning(**tun)
    ws = krex.gemm_workspace()
    for t in range(12):
        M = int(rng.integers(1, 320)) * 8
        N = int(rng.integers(1, 320)) * 8
        K = int(rng.integers(1, 320)) * 8
        if t < 3:
            M, N, K = int(rng.integers(1, 9)) * 8, int(rng.integers(1, 9)) * 8, int(rng.integers(1, 9)) * 8
        seed = 9000 + t
        a, b = _gen(seed, M, N, K)
        c = Guarded(M, N, torch.bfloat16)
        krex.krex_run_candidate_ws(krex.KREX_OP_GEMM_BF16, [a, b], c.view, ws)
        torch.cuda.synchronize()
        assert krex.krex_device_status() == 0 and c.canaries_intact(), (M, N, K)
        ah, bh = gen.uniform_bf16(seed, 0, M, K), gen.uniform_bf16(seed, 1, K, N)
        want = ref.gemm_f64(ah, bh)
        ok, worst = _within_tol(bits16(c.view), want, K)
        assert ok, (M, N, K, worst)
        if not tun:
            # the reference on the same shape: within the fp32 summation bound
            r = Guarded(M, N, torch.float32)
            krex.krex_run_reference(krex.KREX_OP_GEMM_BF16, [a, b], r.view)
            torch.cuda.synchronize()
            assert r.canaries_intact()
            absab = np.abs(gen.bf16_to_f32(ah).astype(np.float64)) @ np.abs(gen.bf16_to_f32(bh).astype(np.float64))
            assert np.all(np.abs(r.view.cpu().numpy() - want) <= (K + 2) * 2.0 ** -24 * absab + 1e-30), (M, N, K)


@pytest.mark.parametrize("ldc_pad", [0, 8, 3])
def test_wide_tiles_output_row_stride(ldc_pad):
    # wide pair tiles (one 512-column accumulator, handed back in halves) with
    # the TMA-store epilogue and, for rows not on 16 bytes, direct stores;
    # several tiles per pair, a ragged last chunk; sentinels intact
    krex.krex_set_tuning(gemm_pair_tile_n=512)
    M, N, K = 2304, 4104, 520
    seed = 4100 + ldc_pad
    a, b = _gen(seed, M, N, K)
    c = Guarded(M, N, torch.bfloat16, ld=N + ldc_pad)
    krex.krex_run_candidate(krex.KREX_OP_GEMM_BF16, [a, b], c.view)
    torch.cuda.synchronize()
    assert krex.krex_device_status() == 0
    assert c.canaries_intact()
    want = ref.gemm_f64(gen.uniform_bf16(seed, 0, M, K), gen.uniform_bf16(seed, 1, K, N))
    ok, worst = _within_tol(bits16(c.view), want, K)
    assert ok, worst


@pytest.mark.parametrize("split", ["0", "1"])
@pytest.mark.parametrize("M,N,K", [(1024, 2048, 512), (4096, 1024, 256), (256, 256, 4096)])
def test_2sm_tail_split_on_and_off(M, N, K, split):
    # a final partial wave of pair tiles is split into column halves (or not)
    krex.krex_set_tuning(gemm_tail_split=int(split))
    seed = 5000 + M + N + K
    a, b = _gen(seed, M, N, K)
    c = _candidate(a, b)
    want = ref.gemm_f64(gen.uniform_bf16(seed, 0, M, K), gen.uniform_bf16(seed, 1, K, N))
    ok, worst = _within_tol(bits16(c), want, K)
    assert ok, worst


def test_k_zero_gives_zero_and_empty_is_noop(variant):
    a = torch.empty(64, 0, dtype=torch.bfloat16, device="cuda")
    b = torch.empty(0, 32, dtype=torch.bfloat16, device="cuda")
    c = torch.full((64, 32), 3.0, dtype=torch.bfloat16, device="cuda")
    krex.krex_run_candidate(krex.KREX_OP_GEMM_BF16, [a, b], c)
    torch.cuda.synchronize()
    assert torch.count_nonzero(c).item() == 0
    e = torch.empty(0, 16, dtype=torch.bfloat16, device="cuda")
    krex.krex_run_candidate(krex.KREX_OP_GEMM_BF16, [e, torch.empty(16, 8, dtype=torch.bfloat16, device="cuda")],
                            torch.empty(0, 8, dtype=torch.bfloat16, device="cuda"))


@pytest.mark.parametrize("lda_pad,ldb_pad", [(8, 0), (0, 16), (24, 40)])
def test_input_row_strides(lda_pad, ldb_pad, variant):
    # A and B as views into wider rows whose padding holds NaN: a kernel that
    # read past a row's K (A) or N (B) elements would put NaN into C.  The
    # reference GEMM gets the same strided operands.
    M, N, K = 300, 1000, 520
    seed = 4100 + lda_pad + ldb_pad
    nan16 = 0x7FC0
    abase = torch.full((M, K + lda_pad), nan16, dtype=torch.int16, device="cuda").view(torch.bfloat16)
    bbase = torch.full((K, N + ldb_pad), nan16, dtype=torch.int16, device="cuda").view(torch.bfloat16)
    a, b = abase[:, :K], bbase[:, :N]
    krex.krex_gen_inputs(seed, 0, krex.KREX_DIST_UNIFORM_PM1, 0.0, a)
    krex.krex_gen_inputs(seed, 1, krex.KREX_DIST_UNIFORM_PM1, 0.0, b)
    c = Guarded(M, N, torch.bfloat16)
    r = Guarded(M, N, torch.float32)
    krex.krex_run_candidate(krex.KREX_OP_GEMM_BF16, [a, b], c.view)
    krex.krex_run_reference(krex.KREX_OP_GEMM_BF16, [a, b], r.view)
    torch.cuda.synchronize()
    assert krex.krex_device_status() == 0
    assert c.canaries_intact() and r.canaries_intact()
    want = ref.gemm_f64(gen.uniform_bf16(seed, 0, M, K), gen.uniform_bf16(seed, 1, K, N))
    ok, worst = _within_tol(bits16(c.view), want, K)
    assert ok, worst
    ok, worst = _within_tol(bits16(r.view.to(torch.bfloat16)), want, K)
    assert ok, worst


def test_unaligned_input_strides_are_rejected():
    # TMA rows must start on 16 bytes: lda or ldb not a multiple of 8 elements
    a = torch.zeros(64, 72, dtype=torch.bfloat16, device="cuda")[:, :64]
    b = torch.zeros(64, 68, dtype=torch.bfloat16, device="cuda")[:, :64]
    c = torch.empty(64, 64, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(krex.KrexError, match="UNSUPPORTED"):
        krex.krex_run_candidate(krex.KREX_OP_GEMM_BF16, [a[:, :60], b[:60]], c)   # K = 60
    a2 = torch.zeros(64 * 68, dtype=torch.bfloat16, device="cuda").view(64, 68)[:, :64]   # lda = 68
    with pytest.raises(krex.KrexError, match="UNSUPPORTED"):
        krex.krex_run_candidate(krex.KREX_OP_GEMM_BF16, [a2, b], c)                # ldb = 68 too


def test_unsupported_shapes_are_rejected():
    a = torch.zeros(16, 12, dtype=torch.bfloat16, device="cuda")
    b = torch.zeros(12, 16, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(krex.KrexError, match="UNSUPPORTED"):
        krex.krex_run_candidate(krex.KREX_OP_GEMM_BF16, [a, b], torch.empty(16, 16, dtype=torch.bfloat16,
                                                                               device="cuda"))


@pytest.mark.parametrize("M,N,K", [(256, 256, 256), (300, 1000, 520), (1024, 2048, 512)])
def test_reference_gemm_within_fp32_bound(M, N, K):
    seed = 77 + M
    a, b = _gen(seed, M, N, K)
    r = Guarded(M, N, torch.float32)
    krex.krex_run_reference(krex.KREX_OP_GEMM_BF16, [a, b], r.view)
    torch.cuda.synchronize()
    assert r.canaries_intact()
    ah, bh = gen.uniform_bf16(seed, 0, M, K), gen.uniform_bf16(seed, 1, K, N)
    want = ref.gemm_f64(ah, bh)
    absab = np.abs(gen.bf16_to_f32(ah).astype(np.float64)) @ np.abs(gen.bf16_to_f32(bh).astype(np.float64))
    # fp32 recursive summation bound: |err| <= K u sum|ab| (u = 2^-24), plus output rounding
    assert np.all(np.abs(r.view.cpu().numpy() - want) <= (K + 2) * 2.0 ** -24 * absab + 1e-30)


def test_gemm_4096_full_output(variant):
    M = N = K = 4096
    a, b = _gen(2, M, N, K)
    c = _candidate(a, b, guard=False)
    want = ref.gemm_f64(gen.uniform_bf16(2, 0, M, K), gen.uniform_bf16(2, 1, K, N))
    ok, worst = _within_tol(bits16(c), want, K)
    assert ok, worst


@pytest.mark.parametrize("n,seed", [(8192, 4), (16384, 5)])
def test_gemm_large_sampled(n, seed):
    a, b = _gen(seed, n, n, n)
    c = _candidate(a, b, guard=False)
    i, j = ref.sample_indices(seed, 2, 4096, n, n)
    got = bits16(c[torch.from_numpy(i).cuda(), torch.from_numpy(j).cuda()])
    want = ref.gemm_sampled_f64(seed, n, n, n, i, j)
    ok, worst = _within_tol(got, want, n)
    assert ok, worst
    # property at any size: the whole output is finite and bounded by K
    assert torch.isfinite(c.float()).all().item()
    assert c.float().abs().max().item() <= n


@pytest.mark.parametrize("ksub", ["2", "1"])
@pytest.mark.parametrize("M,N,K", [(1024, 2048, 512), (256, 256, 4096), (300, 1000, 520), (640, 384, 4104),
                                   (1536, 1536, 3072), (2064, 1000, 1032), (4096, 4096, 256)])
def test_2sm_split_k_tail(M, N, K, ksub):
    # with a workspace the tiles of a GEMM that fits in one partial wave are
    # split into K halves whose fp32 partials meet in the workspace (larger
    # GEMMs keep column halves); two calls in a row (the arrival counters
    # reset themselves, the flags are tagged per launch)
    # the hand-over at every K, not only where it pays
    krex.krex_set_tuning(gemm_stage_k=64 if ksub == "1" else 128, gemm_split_k=1)
    seed = 6000 + M + N + K
    a, b = _gen(seed, M, N, K)
    ws = krex.gemm_workspace()
    want = ref.gemm_f64(gen.uniform_bf16(seed, 0, M, K), gen.uniform_bf16(seed, 1, K, N))
    for _ in range(2):
        c = Guarded(M, N, torch.bfloat16)
        krex.krex_run_candidate_ws(krex.KREX_OP_GEMM_BF16, [a, b], c.view, ws)
        torch.cuda.synchronize()
        assert krex.krex_device_status() == 0
        assert c.canaries_intact()
        ok, worst = _within_tol(bits16(c.view), want, K)
        assert ok, worst
        # the workspace ends with 512 arrival counters, then 512 flags (uint32 each)
        counters = ws[ws.numel() - 4096:ws.numel() - 2048]
        assert torch.count_nonzero(counters).item() == 0  # every arrival counter back at 0


def test_split_k_matches_column_split_closely():
    # K halves and column halves sum the same products in different orders:
    # both within tolerance, and equal in most elements
    krex.krex_set_tuning(gemm_split_k=1)
    M, N, K = 1536, 1536, 3072
    a, b = _gen(2, M, N, K)
    c0 = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    c1 = torch.empty_like(c0)
    krex.krex_run_candidate(krex.KREX_OP_GEMM_BF16, [a, b], c0)
    krex.krex_run_candidate_ws(krex.KREX_OP_GEMM_BF16, [a, b], c1, krex.gemm_workspace())
    torch.cuda.synchronize()
    assert krex.krex_device_status() == 0
    same = (c0.view(torch.int16) == c1.view(torch.int16)).float().mean().item()
    assert same > 0.9
    want = ref.gemm_f64(gen.uniform_bf16(2, 0, M, K), gen.uniform_bf16(2, 1, K, N))
    for c in (c0, c1):
        ok, worst = _within_tol(bits16(c), want, K)
        assert ok, worst


def test_2sm_ragged_edge_items_under_contention():
    # M = N = K = 2064: the last row of pair tiles holds 16 rows, so on its
    # items the second CTA of a pair loads nothing, and one column half lies
    # wholly outside the matrix.  With other kernels sharing the SMs, its
    # producer must still keep step with the leader's MMAs: every launch ends
    # without a time-out and with the right product.
    n = 2064
    a, b = _gen(2064, n, n, n)
    c = torch.empty(n, n, dtype=torch.bfloat16, device="cuda")
    x = torch.empty(16384, 8192, dtype=torch.float32, device="cuda")
    y = torch.empty_like(x)
    krex.krex_gen_inputs(7, 0, krex.KREX_DIST_NORMAL, 2.0, x)
    side = torch.cuda.Stream()
    for _ in range(80):
        krex.krex_run_candidate(krex.KREX_OP_SOFTMAX_F32, [x], y, stream=side)
        krex.krex_run_candidate(krex.KREX_OP_GEMM_BF16, [a, b], c)
    torch.cuda.synchronize()
    detail = krex.krex_device_status_detail()
    try:
        krex.krex_device_status()
    except krex.KrexError as e:
        pytest.fail(f"{e}: {detail}")
    want = ref.gemm_f64(gen.uniform_bf16(2064, 0, n, n), gen.uniform_bf16(2064, 1, n, n))
    ok, worst = _within_tol(bits16(c), want, n)
    assert ok, worst


def test_wide_tiles_ragged_edges_under_contention():
    # the same ragged edges (last row of pair tiles 16 rows high, the last
    # column chunk partly and wholly outside the matrix) with wide tiles,
    # whose accumulator halves change hands on every tile, beside a softmax
    # stream: no wait runs out, and the product is right
    krex.krex_set_tuning(gemm_pair_tile_n=512)
    M, N, K = 2064, 2312, 4128
    a, b = _gen(2065, M, N, K)
    c = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    x = torch.empty(16384, 8192, dtype=torch.float32, device="cuda")
    y = torch.empty_like(x)
    krex.krex_gen_inputs(7, 0, krex.KREX_DIST_NORMAL, 2.0, x)
    side = torch.cuda.Stream()
    for _ in range(40):
        krex.krex_run_candidate(krex.KREX_OP_SOFTMAX_F32, [x], y, stream=side)
        krex.krex_run_candidate(krex.KREX_OP_GEMM_BF16, [a, b], c)
    torch.cuda.synchronize()
    detail = krex.krex_device_status_detail()
    try:
        krex.krex_device_status()
    except krex.KrexError as e:
        pytest.fail(f"{e}: {detail}")
    want = ref.gemm_f64(gen.uniform_bf16(2065, 0, M, K), gen.uniform_bf16(2065, 1, K, N))
    ok, worst = _within_tol(bits16(c), want, K)
    assert ok, worst


# ------------------------------------------------------------- fp16 GEMM ----

def _gen16(seed, M, N, K):
    a = torch.empty(M, K, dtype=torch.float16, device="cuda")
    b = torch.empty(K, N, dtype=torch.float16, device="cuda")
    krex.krex_gen_inputs(seed, 0, krex.KREX_DIST_UNIFORM_PM1, 0.0, a)
    krex.krex_gen_inputs(seed, 1, krex.KREX_DIST_UNIFORM_PM1, 0.0, b)
    return a, b


def _candidate16(a, b, ws=None):
    M, N = a.shape[0], b.shape[1]
    c = Guarded(M, N, torch.float16)
    if ws is None:
        krex.krex_run_candidate(krex.KREX_OP_GEMM_F16, [a, b], c.view)
    else:
        krex.krex_run_candidate_ws(krex.KREX_OP_GEMM_F16, [a, b], c.view, ws)
    torch.cuda.synchronize()
    assert krex.krex_device_status() == 0
    assert c.canaries_intact()
    return c.view


def _within_tol16(got_bits, want64, K):
    got = gen.f16_to_f32(got_bits).astype(np.float64)
    tol = ref.gemm_tolerance(want64, K, dtype="f16")
    err = np.abs(got - want64)
    return np.all(err <= tol), float(np.max(err / tol))


@pytest.mark.parametrize("ksub", ["2", "1"])
def test_f16_identity_and_permutation_are_exact(ksub):
    krex.krex_set_tuning(gemm_stage_k=64 if ksub == "1" else 128)
    a, _ = _gen16(1, 256, 384, 384)
    eye = to_f16_tensor(gen.f32_to_f16(inputs.identity(384).ravel()).reshape(384, 384))
    assert np.array_equal(bits16(_candidate16(a, eye)), bits16(a))
    p, perm = inputs.permutation_matrix(384, 9)
    pt = to_f16_tensor(gen.f32_to_f16(p.ravel()).reshape(384, 384))
    assert np.array_equal(bits16(_candidate16(a, pt)), bits16(a)[:, perm])


def test_f16_small_integers_are_exact():
    # integer products summed exactly in fp32; |C| < 2048 is exact in binary16
    M, N, K = 256, 512, 64
    g = inputs.rng(5)
    a = g.integers(-4, 5, (M, K)).astype(np.float32)
    b = g.integers(-4, 5, (K, N)).astype(np.float32)
    ah, bh = gen.f32_to_f16(a.ravel()).reshape(M, K), gen.f32_to_f16(b.ravel()).reshape(K, N)
    c = _candidate16(to_f16_tensor(ah), to_f16_tensor(bh))
    want = ref.gemm_f64(ah, bh, dtype="f16")
    assert np.array_equal(gen.f16_to_f32(bits16(c)).astype(np.float64), want)


@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (100, 72, 40), (300, 1000, 520), (1024, 2048, 512),
                                   (640, 384, 4104), (2064, 1000, 1032), (4096, 4096, 4096)])
def test_f16_seeded_gemm_within_tolerance(M, N, K):
    krex.krex_set_tuning(gemm_split_k=1)
    seed = 7000 + M + N + K
    a, b = _gen16(seed, M, N, K)
    want = ref.gemm_f64(gen.uniform_f16(seed, 0, M, K), gen.uniform_f16(seed, 1, K, N), dtype="f16")
    for ws in (None, krex.gemm_workspace()):          # column halves / K halves in the tail
        ok, worst = _within_tol16(bits16(_candidate16(a, b, ws)), want, K)
        assert ok, worst


def test_f16_large_sampled():
    n, seed = 8192, 4
    a, b = _gen16(seed, n, n, n)
    c = torch.empty(n, n, dtype=torch.float16, device="cuda")
    krex.krex_run_candidate(krex.KREX_OP_GEMM_F16, [a, b], c)
    torch.cuda.synchronize()
    assert krex.krex_device_status() == 0
    i, j = ref.sample_indices(seed, 2, 4096, n, n)
    got = bits16(c[torch.from_numpy(i).cuda(), torch.from_numpy(j).cuda()])
    want = ref.gemm_sampled_f64(seed, n, n, n, i, j, dtype="f16")
    ok, worst = _within_tol16(got, want, n)
    assert ok, worst


@pytest.mark.parametrize("M,N,K", [(256, 256, 256), (300, 1000, 520)])
def test_f16_reference_gemm_within_fp32_bound(M, N, K):
    seed = 88 + M
    a, b = _gen16(seed, M, N, K)
    r = Guarded(M, N, torch.float32)
    krex.krex_run_reference(krex.KREX_OP_GEMM_F16, [a, b], r.view)
    torch.cuda.synchronize()
    assert r.canaries_intact()
    ah, bh = gen.uniform_f16(seed, 0, M, K), gen.uniform_f16(seed, 1, K, N)
    want = ref.gemm_f64(ah, bh, dtype="f16")
    absab = np.abs(gen.f16_to_f32(ah).astype(np.float64)) @ np.abs(gen.f16_to_f32(bh).astype(np.float64))
    assert np.all(np.abs(r.view.cpu().numpy() - want) <= (K + 2) * 2.0 ** -24 * absab + 1e-30)


def test_f16_op_rejects_bf16_operands():
    a = torch.zeros(16, 16, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(krex.KrexError, match="INVALID"):
        krex.krex_run_candidate(krex.KREX_OP_GEMM_F16, [a, a], torch.empty(16, 16, dtype=torch.float16,
                                                                               device="cuda"))



@pytest.mark.parametrize("f16", [False, True], ids=["bf16", "f16"])
@pytest.mark.parametrize("tile", ["0", "1", "2", "3", "4", "5"])
def test_reference_tilings_are_bit_identical(tile, f16):
    # every output of the reference is one fp32 FMA chain in k order, so the
    # tiling (5: one output per thread, the small-GEMM form) must not change a
    # bit (ragged shape: partial tiles in M, N, K)
    M, N, K = 300, 1000, 520
    a, b = _gen16(99, M, N, K) if f16 else _gen(99, M, N, K)
    op = krex.KREX_OP_GEMM_F16 if f16 else krex.KREX_OP_GEMM_BF16
    r0 = torch.empty(M, N, dtype=torch.float32, device="cuda")
    krex.krex_set_tuning(reference_tiling=0)
    krex.krex_run_reference(op, [a, b], r0)
    r = Guarded(M, N, torch.float32)
    krex.krex_set_tuning(reference_tiling=int(tile))
    krex.krex_run_reference(op, [a, b], r.view)
    torch.cuda.synchronize()
    assert r.canaries_intact()
    assert torch.equal(r.view.contiguous().view(torch.int32), r0.view(torch.int32))


@pytest.mark.parametrize("f16", [False, True], ids=["bf16", "f16"])
def test_reference_unchecked_form_equals_checked_form(f16):
    # a GEMM whose tiles and K slices all lie inside the matrices runs the
    # reference without bounds checks; the same operands with an odd row
    # stride of A (no 16-byte loads) take the checked form: identical bits
    M, N, K = 512, 768, 1024
    a, b = _gen16(77, M, N, K) if f16 else _gen(77, M, N, K)
    op = krex.KREX_OP_GEMM_F16 if f16 else krex.KREX_OP_GEMM_BF16
    r_in = torch.empty(M, N, dtype=torch.float32, device="cuda")
    krex.krex_run_reference(op, [a, b], r_in)
    wide = torch.zeros(M, K + 3, dtype=a.dtype, device="cuda")
    wide[:, :K] = a
    r_chk = Guarded(M, N, torch.float32)
    krex.krex_run_reference(op, [wide[:, :K], b], r_chk.view)
    torch.cuda.synchronize()
    assert r_chk.canaries_intact()
    assert torch.equal(r_chk.view.contiguous().view(torch.int32), r_in.view(torch.int32))


@pytest.mark.parametrize("bn", [256, 512])
@pytest.mark.parametrize("alternate", [0, 1], ids=["forward", "alternating"])
@pytest.mark.parametrize("M,N,K", [(3072, 3072, 4104), (3072, 2560, 200), (4608, 4608, 1032), (4608, 8192, 1032)])
def test_k_direction_alternating_by_wave(M, N, K, alternate, bn):
    # several waves of pair tiles (256 or 512 wide), every other one walking K
    # from its end (a partial last K stage first); forward and alternating
    # orders are both within tolerance, and equal in most elements
    krex.krex_set_tuning(gemm_k_alternate=alternate, gemm_pair_tile_n=bn)
    seed = 8000 + M + N + K
    a, b = _gen(seed, M, N, K)
    c = _candidate(a, b)
    want = ref.gemm_f64(gen.uniform_bf16(seed, 0, M, K), gen.uniform_bf16(seed, 1, K, N))
    ok, worst = _within_tol(bits16(c), want, K)
    assert ok, worst
    if alternate:
        krex.krex_set_tuning(gemm_k_alternate=0, gemm_pair_tile_n=bn)
        c0 = _candidate(a, b)
        same = (c0.view(torch.int16) == c.view(torch.int16)).float().mean().item()
        assert same > 0.5


def test_fma_probe_runs_and_leaves_the_context_clean():
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    sink = torch.zeros(n_sm * 256, dtype=torch.float32, device="cuda")
    krex.krex_probe_fma(256, n_sm, sink)
    torch.cuda.synchronize()
    assert krex.krex_device_status() == 0
    assert torch.count_nonzero(sink).item() == 0     # the sum is never the stored value


@pytest.mark.parametrize("f16", [False, True], ids=["bf16", "f16"])
def test_reference_whole_tile_form_keeps_special_values(f16):
    # the whole-tile reference multiplies 16-bit operands with the mixed-precision
    # FMA; with subnormal operands, signed zeros, infinite operands (inf x 0
    # gives NaN) and (bf16) products that overflow to +-inf it still equals the
    # checked form (operands widened to fp32 first) bit for bit, NaN for NaN
    M, N, K = 640, 640, 64          # 25 tiles of 128 x 128: the tiled (whole-tile) form, not the small one
    g = inputs.rng(11)
    if f16:
        vals = np.array([0.0, -0.0, 2.0 ** -24, -(2.0 ** -20), 2.0 ** -14, 1.0, -2.0, 60000.0, -60000.0],
                        dtype=np.float32)
        enc, dec, tt = gen.f32_to_f16, gen.f16_to_f32, to_f16_tensor
        op = krex.KREX_OP_GEMM_F16
    else:
        vals = np.array([0.0, -0.0, 2.0 ** -130, -(2.0 ** -126), 2.0 ** -133, 1.0, -3.0, 2.0 ** 120, -(2.0 ** 121)],
                        dtype=np.float32)
        enc, dec, tt = gen.f32_to_bf16, gen.bf16_to_f32, to_bf16_tensor
        op = krex.KREX_OP_GEMM_BF16
    a_bits = enc(g.choice(vals, size=M * K)).reshape(M, K)
    b_bits = enc(g.choice(vals, size=K * N)).reshape(K, N)
    assert np.array_equal(dec(enc(vals)), vals)                 # every value is exact in the 16-bit format
    # infinite operands in one row of A and one column of B: inf x 0 = NaN there
    a_bits[3, 5] = enc(np.array([np.inf], dtype=np.float32))[0]
    b_bits[10, 20] = enc(np.array([-np.inf], dtype=np.float32))[0]
    a, b = tt(a_bits), tt(b_bits)
    r_whole = torch.empty(M, N, dtype=torch.float32, device="cuda")
    krex.krex_run_reference(op, [a, b], r_whole)
    wide = torch.zeros(M, K + 3, dtype=a.dtype, device="cuda")
    wide[:, :K] = a
    r_chk = torch.empty(M, N, dtype=torch.float32, device="cuda")
    krex.krex_run_reference(op, [wide[:, :K], b], r_chk)       # odd row stride: the checked form
    torch.cuda.synchronize()
    x, y = r_whole.cpu().numpy(), r_chk.cpu().numpy()
    nan = np.isnan(x)
    assert np.array_equal(nan, np.isnan(y)) and nan.any() and np.isinf(x).any() and np.isfinite(x).any()
    assert np.array_equal(x[~nan].view(np.uint32), y[~nan].view(np.uint32))


@pytest.mark.parametrize("alternate", [0, 1], ids=["forward", "alternating"])
def test_f16_k_direction_alternating_by_wave(alternate):
    krex.krex_set_tuning(gemm_k_alternate=alternate)
    M, N, K = 3072, 3072, 1032
    seed = 8100 + alternate
    a, b = _gen16(seed, M, N, K)
    want = ref.gemm_f64(gen.uniform_f16(seed, 0, M, K), gen.uniform_f16(seed, 1, K, N), dtype="f16")
    ok, worst = _within_tol16(bits16(_candidate16(a, b)), want, K)
    assert ok, worst
