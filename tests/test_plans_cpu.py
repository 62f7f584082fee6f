"""The GEMM, GRU and depthwise-separable planners, run on the host through
the C ABI (isam_gemm_plan_for, isam_gru_plan_for, isam_dwsep_plan_for: host
arithmetic, no CUDA call) with a GB300's limits: 152 SMs, 232448 bytes of
opt-in shared memory per CTA.  Every shape inside the boundary's support
limits (GRU: batch <= 256, hidden any multiple of 32 up to 1024; dwsep: Cin
and Cout multiples of 16 up to 256, any width; GEMM: the benchmark shapes and
a grid of small, ragged and large ones in all four layouts) must get a plan
that fits the device, and the plans must keep the invariants the kernels rely
on."""
import math

import pytest

from paper_1810_09958_gb300 import build, isam

SMS = 152
SMEM = 232448
HIDDEN = list(range(32, 1025, 32))
BATCH = [1, 7, 32, 33, 64, 65, 100, 128, 129, 256]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    isam.load()


def gru_plan(layers, batch, hidden, rb=False):
    return isam.gru_plan(layers, batch, hidden, rb, num_sms=SMS, smem_optin=SMEM)


@pytest.mark.parametrize("layers", [1, 2, 3])
def test_gru_every_supported_shape_has_a_plan_that_fits(layers, monkeypatch):
    monkeypatch.delenv("ISAM_NO_WAVE", raising=False)
    for H in HIDDEN:
        for batch in BATCH:
            for rb in (False, True):
                p = gru_plan(layers, batch, H, rb)
                ks, ka = p["splits"], p["atoms"]
                atoms = math.ceil(H / 64)
                assert ks in (1, 2, 4) and ka == math.ceil(atoms / ks), (H, p)
                # K ranges of whole atoms cover the hidden size, and the last
                # CTA of a cluster still holds part of it.
                assert (ks - 1) * ka * 64 < H <= ks * ka * 64, (H, p)
                assert p["ctas"] == H // 32 * ks <= SMS
                assert 0 < p["smem"] <= SMEM, (H, batch, layers, rb, p)
                bp = p["batch_pad"]
                if batch <= 32:
                    assert bp == 32
                else:
                    assert bp in (64, 128) and (bp == 64 or ks == 4)
                assert p["chunks"] == math.ceil(batch / bp)
                if layers == 1:
                    assert p["path"] == 0
                elif batch > 32:
                    assert p["path"] == 3
                elif not rb and H % 256 == 0:
                    assert p["path"] == 1
                else:
                    assert p["path"] == 2


def test_gru_benchmark_plans():
    """Hidden 1024, batch 32: 32 clusters of 4 CTAs (128), 4 K atoms of U
    each; two stacked layers run as one kernel, the reset-before form as the
    per-layer chain."""
    assert gru_plan(1, 32, 1024) == {"splits": 4, "atoms": 4, "batch_pad": 32, "ctas": 128,
                                     "smem": gru_plan(1, 32, 1024)["smem"], "path": 0, "chunks": 1}
    assert gru_plan(2, 32, 1024)["path"] == 1
    assert gru_plan(2, 32, 1024, rb=True)["path"] == 2
    assert gru_plan(1, 200, 1024)["batch_pad"] == 128 and gru_plan(1, 200, 1024)["chunks"] == 2
    assert gru_plan(1, 64, 1024)["batch_pad"] == 64


def test_gru_uneven_k_ranges():
    """Hidden sizes whose atoms do not divide evenly among the splits."""
    assert (gru_plan(1, 8, 960)["splits"], gru_plan(1, 8, 960)["atoms"]) == (4, 4)   # 15 atoms
    assert (gru_plan(1, 8, 864)["splits"], gru_plan(1, 8, 864)["atoms"]) == (2, 7)   # 13.5 atoms
    assert (gru_plan(1, 8, 448)["splits"], gru_plan(1, 8, 448)["atoms"]) == (1, 7)
    assert (gru_plan(1, 8, 480)["splits"], gru_plan(1, 8, 480)["atoms"]) == (2, 4)


def test_gru_no_wave_switch_selects_the_chain(monkeypatch):
    monkeypatch.setenv("ISAM_NO_WAVE", "1")
    assert gru_plan(2, 32, 1024)["path"] == 2


def test_gru_rejects_shapes_outside_the_limits():
    for (layers, batch, H) in [(1, 257, 64), (1, 1, 80), (1, 1, 1056), (1, 1, 16), (2, 300, 256)]:
        with pytest.raises(isam.IsamError) as e:
            gru_plan(layers, batch, H)
        assert e.value.code == isam.ISAM_ERR_UNSUPPORTED
    # Too few SMs for the co-resident recurrence of hidden 1024 (128 CTAs).
    with pytest.raises(isam.IsamError) as e:
        isam.gru_plan(1, 32, 1024, num_sms=100, smem_optin=SMEM)
    assert e.value.code == isam.ISAM_ERR_UNSUPPORTED
    lib = isam.load()
    import ctypes
    out = (ctypes.c_int * 7)()
    assert lib.isam_gru_plan_for(0, 1, 64, 0, SMS, SMEM, out) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_gru_plan_for(1, 1, 64, 2, SMS, SMEM, out) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_gru_plan_for(1, 1, 64, 0, SMS, SMEM, None) == isam.ISAM_ERR_INVALID_ARG


WIDTHS = [1, 2, 3, 7, 8, 13, 28, 56, 64, 100, 112, 128, 129, 200]


def test_dwsep_every_supported_shape_has_a_plan():
    for W in WIDTHS:
        for cin in range(16, 257, 16):
            for cout in range(16, 257, 16):
                p = isam.dwsep_plan(W, cin, cout, smem_optin=SMEM)
                pc, blocks = p["block_cout"], p["blocks"]
                assert pc % 16 == 0 and 16 <= pc <= cout, (W, cin, cout, p)
                assert blocks == math.ceil(cout / pc) and (blocks - 1) * pc < cout
                if p["kernel"] == 0:
                    rt = p["rows_per_tile"]
                    assert W <= 128 and rt >= 1 and rt * W <= 128, (W, cin, cout, p)
                else:
                    assert p["kernel"] == 1 and p["rows_per_tile"] == 0


def test_dwsep_benchmark_and_wide_layer_plans():
    assert isam.dwsep_plan(56, 128, 256, smem_optin=SMEM) == {"kernel": 0, "rows_per_tile": 2, "blocks": 1,
                                                              "block_cout": 256}
    assert isam.dwsep_plan(56, 256, 256, smem_optin=SMEM) == {"kernel": 1, "rows_per_tile": 0, "blocks": 4,
                                                              "block_cout": 64}
    # More shared memory, fewer blocks: the planner follows the limit it is given.
    assert isam.dwsep_plan(56, 256, 256, smem_optin=400 * 1024)["blocks"] < 4


def test_dwsep_plan_rejects_unsupported_channels():
    for (cin, cout) in [(24, 16), (16, 272), (272, 16), (8, 16)]:
        with pytest.raises(isam.IsamError) as e:
            isam.dwsep_plan(8, cin, cout, smem_optin=SMEM)
        assert e.value.code == isam.ISAM_ERR_UNSUPPORTED
    lib = isam.load()
    import ctypes
    out = (ctypes.c_int * 4)()
    assert lib.isam_dwsep_plan_for(0, 16, 16, SMEM, out) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_dwsep_plan_for(8, 16, 16, SMEM, None) == isam.ISAM_ERR_INVALID_ARG


# ---- the GEMM planner (isam_gemm_plan_for): cluster capacities of 2, 4 and 8
# CTAs as if every SM could hold one CTA of any cluster (the device query can
# only lower them, which the invariants below do not depend on).
CAPS = [SMS // 2, SMS // 4, SMS // 8]


def gemm_plan(M, N, K, tA, tB, beta=0.0, caps=CAPS):
    return isam.gemm_plan(M, N, K, tA, tB, beta, num_sms=SMS, smem_optin=SMEM, cluster_caps=caps)


def check_gemm_plan(M, N, K, tA, tB, p):
    assert p["BN"] in (16, 32, 64, 128, 256), p
    assert p["split"] in (1, 2, 4, 8) and p["cta_pair"] in (1, 2), p
    assert 0 < p["smem"] <= SMEM and 1 <= p["grid"] <= SMS, p
    # Clusters (split-K groups or CTA pairs) fill the grid whole.
    assert p["grid"] % (p["split"] * p["cta_pair"]) == 0, p
    if p["cta_pair"] == 2:
        assert p["tile_m"] == 256 and p["split"] == 1 and tA == 0 and N % 4 == 0 and K >= 256, p
    else:
        assert p["tile_m"] == 128
    # A split never leaves a CTA without K atoms.
    assert p["split"] <= max(1, math.ceil(K / 64)), p


def test_gemm_plans_of_the_benchmark_shapes():
    for (M, K) in [(1760, 1760), (2560, 2560), (4096, 4096), (7680, 2560)]:
        for N in (16, 32, 64, 128):
            for tA in (0, 1):
                check_gemm_plan(M, N, K, tA, 0, gemm_plan(M, N, K, tA, 0))
    p = gemm_plan(8192, 8192, 8192, 0, 0, 1.0)
    check_gemm_plan(8192, 8192, 8192, 0, 0, p)
    assert (p["tile_m"], p["cta_pair"], p["BN"], p["split"]) == (256, 2, 256, 1)
    check_gemm_plan(512, 512, 512, 0, 0, gemm_plan(512, 512, 512, 0, 0))


def test_gemm_plans_over_a_grid_of_shapes():
    sizes = [8, 16, 24, 120, 128, 136, 1000, 2048, 4104]
    for M in sizes:
        for N in sizes:
            for K in sizes:
                for tA in (0, 1):
                    for tB in (0, 1):
                        check_gemm_plan(M, N, K, tA, tB, gemm_plan(M, N, K, tA, tB))


def test_gemm_plans_with_few_resident_clusters():
    for (M, N, K) in [(4096, 16, 4096), (8192, 8192, 8192), (512, 512, 512)]:
        check_gemm_plan(M, N, K, 0, 0, gemm_plan(M, N, K, 0, 0, caps=[1, 1, 1]))


def test_gemm_plan_for_rejects_bad_arguments():
    import ctypes
    lib = isam.load()
    out = (ctypes.c_int * 8)()
    caps = (ctypes.c_int * 3)(*CAPS)
    assert lib.isam_gemm_plan_for(0, 16, 16, 0, 0, 0.0, SMS, SMEM, caps, out) == isam.ISAM_ERR_INVALID_ARG
    assert lib.isam_gemm_plan_for(16, 16, 16, 0, 0, 0.0, SMS, SMEM, None, out) == isam.ISAM_ERR_INVALID_ARG
    zero = (ctypes.c_int * 3)(0, 1, 1)
    assert lib.isam_gemm_plan_for(16, 16, 16, 0, 0, 0.0, SMS, SMEM, zero, out) == isam.ISAM_ERR_INVALID_ARG
    # K = 12: a K-major A row is not 16-byte aligned.
    assert lib.isam_gemm_plan_for(16, 16, 12, 0, 0, 0.0, SMS, SMEM, caps, out) == isam.ISAM_ERR_UNSUPPORTED


def test_gemm_argument_rules_on_the_host():
    """The boundary's GEMM support limits, checked before any CUDA call: sizes
    >= 1, flags 0 or 1, and 16-byte rows of the stored operands (the row pitch
    of A is K when A is M x K, M when it is K x M; of B, N when B is K x N, K
    when it is N x K)."""
    import ctypes
    lib = isam.load()
    out = (ctypes.c_int * 8)()
    caps = (ctypes.c_int * 3)(*CAPS)
    cases = [
        ((16, 16, 16, 0, 0), isam.ISAM_OK),
        ((16, 16, 16, 1, 1), isam.ISAM_OK),
        ((13, 16, 16, 0, 0), isam.ISAM_OK),                 # M free when A is M x K
        ((13, 16, 16, 1, 0), isam.ISAM_ERR_UNSUPPORTED),    # A stored K x 13: 26-byte rows
        ((16, 13, 16, 0, 1), isam.ISAM_OK),                 # N free when B is N x K
        ((16, 13, 16, 0, 0), isam.ISAM_ERR_UNSUPPORTED),    # B stored K x 13
        ((16, 16, 12, 0, 1), isam.ISAM_ERR_UNSUPPORTED),    # K-major rows of 24 bytes
        ((16, 16, 12, 1, 0), isam.ISAM_OK),                 # K is only a row count here
        ((1, 1, 8, 0, 1), isam.ISAM_OK),
        ((0, 16, 16, 0, 0), isam.ISAM_ERR_INVALID_ARG),
        ((16, 16, 16, 2, 0), isam.ISAM_ERR_INVALID_ARG),
        ((16, 16, 16, 0, -1), isam.ISAM_ERR_INVALID_ARG),
    ]
    for (M, N, K, tA, tB), want in cases:
        got = lib.isam_gemm_plan_for(M, N, K, tA, tB, 0.0, SMS, SMEM, caps, out)
        assert got == want, ((M, N, K, tA, tB), got, isam.last_error())
