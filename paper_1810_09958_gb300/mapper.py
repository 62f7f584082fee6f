"""Loop-nest -> GEMM mapper (host side): which isam_gemm call computes a kernel.

A restatement of the paper's instruction mapping (Section 2) for the one
instruction this library exposes, a matrix multiplication:

* Programs are written in three-operand form (ISAMIR, Section 2.1): every
  statement performs one operation over the whole loop domain, and buffer
  indices are affine in the loop axes.
* Each buffer access is an *access matrix*: buffer dimensions on the rows,
  loop axes on the columns (Section 2.2).  Mapping a program (the "haystack")
  onto the matmul instruction (the "needle") means choosing an axis map and,
  per buffer, a dimension map such that the selected sub-matrices of the
  haystack equal the needle's.  The search is a recursive backtracking over
  axes with early rejection, as the paper describes.
* When the statement sequence does not match (the separable depthwise
  convolution carries a second multiplication inside the sum), the
  deterministic mapper reports where and why it failed, and the factorisation
  pass (Section 2.3) pulls the factor that does not use the inner reduction
  axes out of that sum, leaving a stage the mapper accepts.  An axis-fusion
  pass merges axes that always appear together as one contiguous index (the
  batch and spatial axes of an NHWC tensor), so the GEMM has a single M.

The result names the isam_gemm arguments (M, N, K, transA, transB), the axes
left outside the instruction (a loop of calls), and the buffers whose mapped
dimensions are not a packed row-major slice (they need a transpose first, as
the paper's mapped 1-D convolution shows).  Nothing here runs on the GPU.

Program text::

    forall i:4, j:3, k:5 {
      tmp[i][j][k] := A[i][k];
      tmp[i][j][k] *= B[k][j];
      C[i][j] += tmp[i][j][k];
    }

Index expressions are affine: ``x+d``, ``2*i+di-1``.
"""
from __future__ import annotations

import itertools
import re
from dataclasses import dataclass, field

import numpy as np

# --------------------------------------------------------------------------- IR


@dataclass(frozen=True)
class Access:
    """buffer[row_0][row_1]...: each row maps axis -> integer coefficient,
    plus a constant offset."""
    buffer: str
    rows: tuple  # tuple of (tuple of (axis, coef) sorted, offset)

    def coef(self, dim: int, axis: str) -> int:
        return dict(self.rows[dim][0]).get(axis, 0)

    def axes(self) -> set:
        return {a for terms, _ in self.rows for a, c in terms if c}

    def row_axes(self, dim: int) -> set:
        return {a for a, c in self.rows[dim][0] if c}


@dataclass(frozen=True)
class Stmt:
    op: str        # ':=', '*=' or '+='
    target: Access
    source: Access


@dataclass
class Program:
    axes: dict     # axis -> extent, in declaration order
    stmts: list

    def buffers(self) -> set:
        return {s.source.buffer for s in self.stmts} | {s.target.buffer for s in self.stmts}


_TERM = re.compile(r"\s*([+-]?)\s*(?:(\d+)\s*\*\s*)?([A-Za-z_][A-Za-z_0-9]*|\d+)\s*")


def _parse_index(expr: str, axes: dict) -> tuple:
    terms, off = {}, 0
    pos = 0
    expr = expr.strip()
    while pos < len(expr):
        m = _TERM.match(expr, pos)
        if not m or m.end() == pos:
            raise ValueError(f"cannot parse index '{expr}'")
        sign = -1 if m.group(1) == "-" else 1
        mult = int(m.group(2)) if m.group(2) else 1
        name = m.group(3)
        if name.isdigit():
            off += sign * mult * int(name)
        else:
            if name not in axes:
                raise ValueError(f"unknown axis '{name}' in '{expr}'")
            terms[name] = terms.get(name, 0) + sign * mult
        pos = m.end()
    return tuple(sorted((a, c) for a, c in terms.items() if c)), off


def _parse_access(text: str, axes: dict) -> Access:
    m = re.fullmatch(r"\s*([A-Za-z_][A-Za-z_0-9]*)\s*((?:\[[^\]]*\])+)\s*", text)
    if not m:
        raise ValueError(f"cannot parse access '{text}'")
    idx = re.findall(r"\[([^\]]*)\]", m.group(2))
    return Access(m.group(1), tuple(_parse_index(e, axes) for e in idx))


def parse(text: str) -> Program:
    """Parses the ISAMIR subset shown in the module docstring."""
    m = re.search(r"forall\s+(.*?)\{(.*)\}", text, re.S)
    if not m:
        raise ValueError("expected 'forall axes { statements }'")
    axes = {}
    for part in m.group(1).split(","):
        name, _, ext = part.strip().partition(":")
        axes[name.strip()] = int(ext)
    stmts = []
    for line in m.group(2).split(";"):
        line = line.strip()
        if not line:
            continue
        lm = re.fullmatch(r"(.+?)\s*(:=|\*=|\+=)\s*(.+)", line)
        if not lm:
            raise ValueError(f"cannot parse statement '{line}'")
        stmts.append(Stmt(lm.group(2), _parse_access(lm.group(1), axes), _parse_access(lm.group(3), axes)))
    return Program(axes, stmts)


def evaluate(prog: Program, buffers: dict) -> dict:
    """Runs the program statement by statement over its whole domain (the IR's
    semantics, Section 2.1) in float64; returns every buffer written.  Indices
    outside a source buffer read zero (zero padding)."""
    env = {k: np.asarray(v, dtype=np.float64) for k, v in buffers.items()}
    names = list(prog.axes)
    grids = np.meshgrid(*[np.arange(prog.axes[a]) for a in names], indexing="ij")
    ax = dict(zip(names, grids))

    def index(acc: Access):
        return [sum((c * ax[a] for a, c in terms), np.zeros_like(grids[0])) + off for terms, off in acc.rows]

    for st in prog.stmts:
        src = env[st.source.buffer]
        idx = index(st.source)
        ok = np.ones(grids[0].shape, dtype=bool)
        for d, i in enumerate(idx):
            ok &= (i >= 0) & (i < src.shape[d])
        val = np.where(ok, src[tuple(np.clip(i, 0, src.shape[d] - 1) for d, i in enumerate(idx))], 0.0)
        tidx = index(st.target)
        if st.target.buffer not in env:
            shape = tuple(int(i.max()) + 1 for i in tidx)
            env[st.target.buffer] = np.zeros(shape)
        tgt = env[st.target.buffer]
        key = tuple(tidx)
        if st.op == ":=":
            tgt[key] = val
        elif st.op == "*=":
            tgt[key] = tgt[key] * val
        else:  # '+=': every domain point adds its value (a reduction where axes are missing)
            np.add.at(tgt, key, val)
    return env


# --------------------------------------------------------------------------- the needle

NEEDLE = parse("""
forall i:1, j:1, k:1 {
  tmp[i][j][k] := A[i][k];
  tmp[i][j][k] *= B[k][j];
  C[i][j] += tmp[i][j][k];
}""")


class MapFailure(Exception):
    """The deterministic mapper's feedback: which statement did not match."""

    def __init__(self, stmt: int, reason: str):
        super().__init__(f"statement {stmt}: {reason}")
        self.stmt = stmt
        self.reason = reason


@dataclass
class GemmMapping:
    """One isam_gemm call (per point of the outer axes)."""
    M: int
    N: int
    K: int
    transA: int
    transB: int
    A: str
    B: str
    C: str
    axis_map: dict           # needle axis (i, j, k) -> haystack axis
    dim_maps: dict           # needle buffer -> {needle dim: haystack dim}
    outer_axes: list         # haystack axes looped around the call
    transposes: dict = field(default_factory=dict)  # buffer -> permutation that packs it

    @property
    def degenerate(self) -> bool:
        """A matrix-vector (or smaller) product: M, N or K is 1."""
        return min(self.M, self.N, self.K) == 1


def _roles(prog: Program):
    ops = [s.op for s in prog.stmts]
    want = [":=", "*=", "+="]
    for n, (got, exp) in enumerate(zip(ops, want)):
        if got != exp:
            raise MapFailure(n, f"operation '{got}' where the matmul has '{exp}'")
    if len(ops) != 3:
        raise MapFailure(min(len(ops), 3), f"{len(ops)} statements where the matmul has 3")
    s0, s1, s2 = prog.stmts
    if not (s0.target == s1.target == s2.source):
        raise MapFailure(2, "the reduction does not consume the product's temporary")
    return s0.source, s1.source, s2.target


def _dim_map(hay: Access, needle: Access, phi: dict):
    """Needle dims -> distinct haystack dims with equal coefficients on the
    mapped axes; unselected haystack dims must not use a mapped axis."""
    mapped = set(phi.values())
    cands = []
    for r in range(len(needle.rows)):
        want = {phi[a]: c for a, c in needle.rows[r][0]}
        opts = [d for d in range(len(hay.rows))
                if {a: c for a, c in hay.rows[d][0] if a in mapped} == want]
        if not opts:
            return None
        cands.append(opts)
    for choice in itertools.product(*cands):
        if len(set(choice)) != len(choice):
            continue
        rest = set(range(len(hay.rows))) - set(choice)
        if any(hay.row_axes(d) & mapped for d in rest):
            continue
        return dict(enumerate(choice))
    return None


def _packing(acc: Access, dims: list) -> list | None:
    """Permutation of acc's dims putting `dims` (in this order) innermost, or
    None when they already are."""
    n = len(acc.rows)
    if list(range(n - len(dims), n)) == list(dims):
        return None
    rest = [d for d in range(n) if d not in dims]
    return rest + list(dims)


def map_matmul(prog: Program) -> GemmMapping:
    """The deterministic mapper: raises MapFailure with feedback when the
    program is not (a loop of) matrix multiplications."""
    x, y, c = _roles(prog)
    red = [a for a in prog.axes if a not in c.axes()]
    best, best_key = None, None
    for a_acc, b_acc in ((x, y), (y, x)):  # the product commutes
        # Recursive search over (i, j, k) with early pruning by axis usage.
        for k in red:
            if k not in a_acc.axes() or k not in b_acc.axes():
                continue
            for i in prog.axes:
                if i == k or i not in a_acc.axes() or i not in c.axes() or i in b_acc.axes():
                    continue
                for j in prog.axes:
                    if j in (i, k) or j not in b_acc.axes() or j not in c.axes() or j in a_acc.axes():
                        continue
                    phi = {"i": i, "j": j, "k": k}
                    dms = {}
                    for nb, hb in (("A", a_acc), ("B", b_acc), ("C", c)):
                        nacc = {"A": NEEDLE.stmts[0].source, "B": NEEDLE.stmts[1].source,
                                "C": NEEDLE.stmts[2].target}[nb]
                        dm = _dim_map(hb, nacc, phi)
                        if dm is None:
                            break
                        dms[nb] = dm
                    else:
                        cand = _build(prog, phi, dms, a_acc, b_acc, c)
                        # Prefer the most work per call, then the fewest transposes.
                        key = (-(cand.M * cand.N * cand.K), len(cand.transposes))
                        if best is None or key < best_key:
                            best, best_key = cand, key
    if best is None:
        raise MapFailure(2, "no axis and dimension map makes the accesses those of a matmul")
    return best


def _build(prog, phi, dms, a_acc, b_acc, c) -> GemmMapping:
    ext = prog.axes
    transA = 0 if dms["A"][0] < dms["A"][1] else 1      # (i, k): i major -> M x K
    transB = 0 if dms["B"][0] < dms["B"][1] else 1      # (k, j): k major -> K x N
    transposes = {}
    for nb, acc in (("A", a_acc), ("B", b_acc), ("C", c)):
        dims = sorted(dms[nb].values())
        perm = _packing(acc, dims)
        if perm is not None:
            transposes[acc.buffer] = perm
    # C must be row-major M x N for the library: compute C^T = B^T A^T otherwise.
    if dms["C"][0] > dms["C"][1]:
        phi = {"i": phi["j"], "j": phi["i"], "k": phi["k"]}
        a_acc, b_acc = b_acc, a_acc
        transA, transB = 1 - transB, 1 - transA
        dms = {"A": {0: dms["B"][1], 1: dms["B"][0]}, "B": {0: dms["A"][1], 1: dms["A"][0]},
               "C": {0: dms["C"][1], 1: dms["C"][0]}}
    outer = [a for a in prog.axes if a not in phi.values()]
    return GemmMapping(M=ext[phi["i"]], N=ext[phi["j"]], K=ext[phi["k"]], transA=transA, transB=transB,
                       A=a_acc.buffer, B=b_acc.buffer, C=c.buffer, axis_map=phi, dim_maps=dms,
                       outer_axes=outer, transposes=transposes)


# --------------------------------------------------------------------------- transformations


def factorize(prog: Program) -> tuple[Program, Program]:
    """Factorisation pass (Section 2.3) for  C += X * Y * F  where the factor F
    does not use some reduction axes R:  C += (sum over R of X * Y) * F.
    Returns stage 1 (T += X * Y, summing over R) and stage 2
    (tmp := T; tmp *= F; C += tmp).  T is indexed by the axes X and Y use
    other than R, in the program's axis order."""
    ops = [s.op for s in prog.stmts]
    if ops != [":=", "*=", "*=", "+="]:
        raise MapFailure(0, "factorisation expects := *= *= +=")
    s0, s1, s2, s3 = prog.stmts
    c = s3.target
    red = [a for a in prog.axes if a not in c.axes()]
    for fac, keep in ((s2.source, s1.source), (s1.source, s2.source)):
        inner = [a for a in red if a not in fac.axes()]
        if not inner:
            continue
        used = s0.source.axes() | keep.axes()
        t_axes = [a for a in prog.axes if a in used and a not in inner]
        t_acc = Access("T", tuple((((a, 1),), 0) for a in t_axes))
        stage1_axes = {a: e for a, e in prog.axes.items() if a in used}
        tmp1 = Access("tmp1", tuple((((a, 1),), 0) for a in stage1_axes))
        stage1 = Program(stage1_axes, [Stmt(":=", tmp1, s0.source), Stmt("*=", tmp1, keep),
                                       Stmt("+=", t_acc, tmp1)])
        stage2_axes = {a: e for a, e in prog.axes.items() if a not in inner}
        tmp2 = Access("tmp2", tuple((((a, 1),), 0) for a in stage2_axes))
        stage2 = Program(stage2_axes, [Stmt(":=", tmp2, t_acc), Stmt("*=", tmp2, fac), Stmt("+=", c, tmp2)])
        return stage1, stage2
    raise MapFailure(2, "no factor is independent of a reduction axis")


def fuse_axes(prog: Program, outer: str, inner: str) -> Program | None:
    """Merges axes (outer, inner) into one axis of extent outer*inner when every
    access either uses neither or addresses them as one contiguous index:
    adjacent dims [.. outer][inner ..] with unit coefficients, or a single dim
    ext(inner)*outer + inner.  Returns None when they cannot be fused."""
    e_in = prog.axes[inner]
    name = f"{outer}{inner}"
    new_stmts = []

    def fuse_acc(acc: Access):
        rows = list(acc.rows)
        uses = [acc.coef(d, outer) or acc.coef(d, inner) for d in range(len(rows))]
        dims_o = [d for d in range(len(rows)) if acc.coef(d, outer)]
        dims_i = [d for d in range(len(rows)) if acc.coef(d, inner)]
        if not dims_o and not dims_i:
            return acc
        if len(dims_o) != 1 or len(dims_i) != 1:
            return None
        do, di = dims_o[0], dims_i[0]
        if do == di:  # one dim: e_in*outer + inner
            terms = dict(rows[do][0])
            if terms[outer] != e_in or terms[inner] != 1:
                return None
            terms.pop(outer)
            terms.pop(inner)
            terms[name] = 1
            rows[do] = (tuple(sorted(terms.items())), rows[do][1])
            return Access(acc.buffer, tuple(rows))
        if di != do + 1:
            return None
        to, ti = dict(rows[do][0]), dict(rows[di][0])
        if to != {outer: 1} or ti != {inner: 1} or rows[do][1] or rows[di][1]:
            return None
        rows[do] = (((name, 1),), 0)
        del rows[di]
        return Access(acc.buffer, tuple(rows))

    for st in prog.stmts:
        t, s = fuse_acc(st.target), fuse_acc(st.source)
        if t is None or s is None:
            return None
        new_stmts.append(Stmt(st.op, t, s))
    axes = {}
    for a, e in prog.axes.items():
        if a == outer:
            axes[name] = e * e_in
        elif a != inner:
            axes[a] = e
    return Program(axes, new_stmts)


def fuse_all(prog: Program) -> Program:
    """Applies axis fusion until no adjacent pair of axes can be fused."""
    changed = True
    while changed:
        changed = False
        names = list(prog.axes)
        for o, i in itertools.permutations(names, 2):
            f = fuse_axes(prog, o, i)
            if f is not None:
                prog, changed = f, True
                break
    return prog


def map_program(prog: Program) -> list:
    """The non-deterministic mapper in the small: try the deterministic mapper;
    on the feedback "a second multiplication where the reduction should be",
    factorise and map each stage.  Returns a list of (stage program after axis
    fusion, GemmMapping or None); a stage whose best mapping is degenerate
    (matrix-vector) keeps it but says so through GemmMapping.degenerate."""
    try:
        fused = fuse_all(prog)
        return [(fused, map_matmul(fused))]
    except MapFailure as f:
        if f.stmt == 2 and "'*='" in f.reason:
            out = []
            for st in factorize(prog):
                fused = fuse_all(st)
                try:
                    out.append((fused, map_matmul(fused)))
                except MapFailure:
                    out.append((fused, None))
            return out
        raise
