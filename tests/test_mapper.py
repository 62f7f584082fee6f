"""The loop-nest -> GEMM mapper (Section 2) on the paper's listings: each
emitted call is executed (numpy, and on the GPU through isam_gemm) and
compared with the loop nest itself evaluated statement by statement."""
import itertools

import numpy as np
import pytest

from paper_1810_09958_gb300 import mapper as mp

MATMUL = """forall i:7, j:5, k:6 {
  tmp[i][j][k] := A[i][k];
  tmp[i][j][k] *= B[k][j];
  C[i][j] += tmp[i][j][k]; }"""


def rand_buffers(prog, names, rng, shapes):
    return {n: rng.integers(-3, 4, size=shapes[n]).astype(np.float64) for n in names}


def execute(prog, m, bufs, out_shape):
    """Runs the mapping's calls: for every point of the outer axes, slice A, B
    and C along the mapped dimensions (the other dimensions are fixed by the
    outer axes), multiply, accumulate."""
    out = np.zeros(out_shape)
    accs = {}
    for st in prog.stmts:
        accs.setdefault(st.source.buffer, st.source)
        accs.setdefault(st.target.buffer, st.target)
    ext = prog.axes
    needle_axes = {"A": ("i", "k"), "B": ("k", "j"), "C": ("i", "j")}

    def view(name, role, env, vals):
        acc = accs[name]
        dm = m.dim_maps[role]
        idx = []
        mapped_dims = {dm[0]: needle_axes[role][0], dm[1]: needle_axes[role][1]}
        for d, (terms, off) in enumerate(acc.rows):
            base = off + sum(c * vals.get(a, 0) for a, c in terms if a not in m.axis_map.values())
            if d in mapped_dims:
                idx.append(slice(base, base + ext[m.axis_map[mapped_dims[d]]]))
            else:
                idx.append(base)
        return idx

    for point in itertools.product(*[range(ext[a]) for a in m.outer_axes]):
        vals = dict(zip(m.outer_axes, point))
        a_idx = view(m.A, "A", bufs, vals)
        b_idx = view(m.B, "B", bufs, vals)
        c_idx = view(m.C, "C", bufs, vals)
        a = bufs[m.A][tuple(a_idx)]
        b = bufs[m.B][tuple(b_idx)]
        # the slices come out in the buffer's dim order: bring them to (i, k) and (k, j)
        if m.dim_maps["A"][0] > m.dim_maps["A"][1]:
            a = a.T
        if m.dim_maps["B"][0] > m.dim_maps["B"][1]:
            b = b.T
        prod = a @ b
        if m.dim_maps["C"][0] > m.dim_maps["C"][1]:
            prod = prod.T
        out[tuple(c_idx)] += prod
    return out


def check(text, shapes, out_name, out_shape, seed=0):
    prog = mp.parse(text)
    m = mp.map_matmul(prog)
    rng = np.random.default_rng(seed)
    bufs = rand_buffers(prog, shapes.keys(), rng, shapes)
    ref = mp.evaluate(prog, dict(bufs, **{out_name: np.zeros(out_shape)}))[out_name]
    got = execute(prog, m, bufs, out_shape)
    assert np.array_equal(got, ref)
    return m


def test_matmul_listing_maps_to_itself():
    m = check(MATMUL, {"A": (7, 6), "B": (6, 5)}, "C", (7, 5))
    assert (m.M, m.N, m.K, m.transA, m.transB) == (7, 5, 6, 0, 0)
    assert m.axis_map == {"i": "i", "j": "j", "k": "k"} and m.outer_axes == [] and not m.transposes


def test_loop_order_and_buffer_transposition_do_not_matter():
    """Reordered loops, A stored K x M and B stored N x K: the same GEMM with
    both operands transposed (Section 2: robust to reordering/transposition)."""
    text = """forall k:6, j:5, i:7 {
      tmp[i][j][k] := A[k][i];
      tmp[i][j][k] *= B[j][k];
      C[i][j] += tmp[i][j][k]; }"""
    m = check(text, {"A": (6, 7), "B": (5, 6)}, "C", (7, 5), seed=1)
    assert (m.M, m.N, m.K, m.transA, m.transB) == (7, 5, 6, 1, 1)


def test_transposed_output_swaps_the_operands():
    """C stored N x M: the library writes row-major C, so the call computes
    C^T = B^T A^T (operands swapped, transposes flipped)."""
    text = """forall i:7, j:5, k:6 {
      tmp[i][j][k] := A[i][k];
      tmp[i][j][k] *= B[k][j];
      Ct[j][i] += tmp[i][j][k]; }"""
    prog = mp.parse(text)
    m = mp.map_matmul(prog)
    assert (m.A, m.B, m.M, m.N, m.K) == ("B", "A", 5, 7, 6)
    assert (m.transA, m.transB) == (1, 1)
    rng = np.random.default_rng(2)
    A, B = rng.integers(-3, 4, (7, 6)).astype(float), rng.integers(-3, 4, (6, 5)).astype(float)
    ref = mp.evaluate(prog, {"A": A, "B": B, "Ct": np.zeros((5, 7))})["Ct"]
    # isam_gemm semantics: C = op(A) op(B), op(X) = X^T when trans.
    opA = B.T if m.transA else B
    opB = A.T if m.transB else A
    assert np.array_equal(opA @ opB, ref)


def test_1d_convolution_listing():
    """The 1-D convolution maps onto a loop of matmuls over the outer axes."""
    text = """forall i:2, x:6, d:3, ki:4, ko:5 {
      tmp[i][x][d][ki][ko] := A[i][x+d][ki];
      tmp[i][x][d][ki][ko] *= B[d][ki][ko];
      C[i][x][ko] += tmp[i][x][d][ki][ko]; }"""
    m = check(text, {"A": (2, 8, 4), "B": (3, 4, 5)}, "C", (2, 6, 5), seed=3)
    assert m.K == 4 and m.axis_map["k"] == "ki" and m.axis_map["j"] == "ko"
    assert set(m.outer_axes) == {"i", "d"}


def test_transpose_reported_when_mapped_dims_are_not_innermost():
    text = """forall i:4, j:3, k:5, b:2 {
      tmp[i][j][k][b] := A[i][b][k];
      tmp[i][j][k][b] *= B[b][k][j];
      C[b][i][j] += tmp[i][j][k][b]; }"""
    m = check(text, {"A": (4, 2, 5), "B": (2, 5, 3)}, "C", (2, 4, 3), seed=4)
    assert m.outer_axes == ["b"]
    assert m.transposes == {"A": [1, 0, 2]}


DWSEP = """forall b:2, i:5, j:6, k:8, di:3, dj:3, q:4, r:1 {
  tmp[b][i][j][k][di][dj][q][r] := X[b][i+di-1][j+dj-1][q];
  tmp[b][i][j][k][di][dj][q][r] *= D[di][dj][q][r];
  tmp[b][i][j][k][di][dj][q][r] *= P[q+r][k];
  C[b][i][j][k] += tmp[b][i][j][k][di][dj][q][r]; }"""


def test_separable_depthwise_needs_factorisation():
    """The extra multiplication stops the deterministic mapper at statement 2;
    factorising P out of the window sum leaves the pointwise stage, which is
    the isam_dwsep_conv GEMM: M = N*H*W, N = Cout, K = Cin, NN."""
    prog = mp.parse(DWSEP)
    with pytest.raises(mp.MapFailure) as e:
        mp.map_matmul(prog)
    assert e.value.stmt == 2 and "'*='" in e.value.reason
    (s1, m1), (s2, m2) = mp.map_program(prog)
    assert m1 is None or m1.degenerate            # the window sum is no GEMM
    assert (m2.M, m2.N, m2.K, m2.transA, m2.transB) == (2 * 5 * 6, 8, 4, 0, 0)
    assert not m2.transposes and not m2.outer_axes
    # The two stages compute the original program.
    rng = np.random.default_rng(5)
    bufs = {"X": rng.integers(-3, 4, (2, 5, 6, 4)).astype(float),
            "D": rng.integers(-3, 4, (3, 3, 4, 1)).astype(float),
            "P": rng.integers(-3, 4, (4, 8)).astype(float)}
    ref = mp.evaluate(prog, dict(bufs, C=np.zeros((2, 5, 6, 8))))["C"]
    st1, st2 = mp.factorize(prog)
    T = mp.evaluate(st1, dict(bufs, T=np.zeros((2, 5, 6, 4, 1))))["T"]
    got = T.reshape(m2.M, m2.K) @ bufs["P"].reshape(m2.K, m2.N)
    assert np.array_equal(got.reshape(2, 5, 6, 8), ref)


GRU_PROJ = """forall t:3, b:2, g:12, h:4 {
  tmp[t][b][g][h] := X[t][b][h];
  tmp[t][b][g][h] *= W[g][h];
  G[t][b][g] += tmp[t][b][g][h]; }"""


def test_gru_input_projection_is_one_gemm():
    """x [T][B][H] times W^T ([3H][H] stored): M = T*B, N = 3H, K = H, B
    transposed -- the call isam_gru_forward makes for its projection."""
    (st, m), = mp.map_program(mp.parse(GRU_PROJ))
    assert (m.M, m.N, m.K, m.transA, m.transB) == (6, 12, 4, 0, 1)
    assert (m.A, m.B, m.C) == ("X", "W", "G")


def test_elementwise_product_is_not_a_matmul():
    text = """forall i:4, j:3 {
      tmp[i][j] := A[i][j];
      tmp[i][j] *= B[i][j];
      C[i][j] += tmp[i][j]; }"""
    with pytest.raises(mp.MapFailure):
        mp.map_matmul(mp.parse(text))


def test_axis_fusion_needs_contiguous_indices():
    prog = mp.parse(GRU_PROJ)
    assert mp.fuse_axes(prog, "t", "b") is not None
    assert mp.fuse_axes(prog, "b", "t") is None      # b is not the outer of the pair
    assert mp.fuse_axes(prog, "g", "h") is None      # used in different accesses


@pytest.mark.gpu
def test_emitted_calls_run_through_isam_gemm():
    """The GRU projection and the depthwise-separable pointwise stage, mapped
    at small sizes, executed by isam_gemm with the emitted arguments."""
    import torch
    from paper_1810_09958_gb300 import build, isam, synth
    from gpu_util import dev_bf16, nmax_err
    build.build()
    isam.load()
    torch.cuda.set_device(0)
    T, B, H = 4, 8, 64
    text = GRU_PROJ.replace("t:3", f"t:{T}").replace("b:2", f"b:{B}").replace("g:12", f"g:{3 * H}").replace(
        "h:4", f"h:{H}")
    prog = mp.parse(text)
    (_, m), = mp.map_program(prog)
    X = synth.bf16_uniform(11, (T, B, H))
    W = synth.bf16_uniform(12, (3 * H, H))
    ref = mp.evaluate(prog, {"X": synth.bf16_bits_to_f64(X), "W": synth.bf16_bits_to_f64(W),
                             "G": np.zeros((T, B, 3 * H))})["G"]
    C = torch.zeros(m.M * m.N, dtype=torch.float32, device="cuda")
    isam.gemm(m.M, m.N, m.K, m.transA, m.transB, 1.0, dev_bf16(X), dev_bf16(W), 0.0, C)
    isam.sync()
    assert nmax_err(C.cpu().numpy().reshape(T, B, 3 * H), ref) <= 5e-3
    # Pointwise stage of the separable layer: T (the window sums) times P.
    Nn, Hh, Ww, Cin, Cout = 2, 5, 6, 64, 48
    text = (DWSEP.replace("b:2", f"b:{Nn}").replace("i:5", f"i:{Hh}").replace("j:6", f"j:{Ww}")
            .replace("k:8", f"k:{Cout}").replace("q:4", f"q:{Cin}"))
    (_, _), (_, m2) = mp.map_program(mp.parse(text))
    Tm = synth.bf16_uniform(13, (Nn, Hh, Ww, Cin))
    P = synth.bf16_uniform(14, (Cin, Cout))
    ref2 = synth.bf16_bits_to_f64(Tm).reshape(-1, Cin) @ synth.bf16_bits_to_f64(P)
    C2 = torch.zeros(m2.M * m2.N, dtype=torch.float32, device="cuda")
    isam.gemm(m2.M, m2.N, m2.K, m2.transA, m2.transB, 1.0, dev_bf16(Tm), dev_bf16(P), 0.0, C2)
    isam.sync()
    assert nmax_err(C2.cpu().numpy().reshape(m2.M, m2.N), ref2) <= 5e-3
