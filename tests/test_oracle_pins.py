"""Pins for the CPU oracle against what the paper and the mathematics fix.

Every check here is independent of the oracle's own code path: hand-derived trees from
the paper's step equations (tests/golden/trees.txt), the paper's closed-form traffic
and computation counts, the definition of Allreduce for integer and max/min cases, the
standard floating-point summation error bound, and a library routine for bf16
rounding.  The last group plants plausible mistakes in the oracle and checks that the
pins catch them.
"""

import os

import numpy as np
import pytest
import torch

import oracle
from oracle import gar_oracle as G

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "trees.txt")


def _golden():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            kind, P, S, p, tree = line.split(None, 4)
            rows.append((kind, int(P), int(S), int(p), G.parse_tree(tree)))
    return rows


def _mpi_partition(n, P):
    """Block boundaries written out here, independently of the oracle: MPI
    reduce_scatter's split, where the first n mod P blocks are one element longer
    (reading C3 of the paper's u = m/P, Sec. "Communication model", eq. initial_data)."""
    q, rem = n // P, n % P
    starts = [i * q + min(i, rem) for i in range(P + 1)]
    return [(starts[i], starts[i + 1]) for i in range(P)]


def _Ls(P):
    L = G.ceil_log2(P)
    return L, list(range(L, 2 * L + 1))


# ---------------------------------------------------------------------------
# Worked trees (hand-derived from eqs. bo_step_even / bo_step_odd / shifted forms)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("row", _golden(), ids=lambda r: f"{r[0]}-P{r[1]}-S{r[2]}-p{r[3]}")
def test_golden_tree(row):
    kind, P, S, p, tree = row
    run = G.simulate(P, 0, S)
    key = run.after_reduction[p]
    assert key[0] == p
    assert run.exprs.tree(key[1]) == tree


@pytest.mark.parametrize("row", _golden(), ids=lambda r: f"{r[0]}-P{r[1]}-S{r[2]}-p{r[3]}")
def test_golden_tree_values(row):
    """The oracle's float32 arithmetic follows the hand-derived tree: evaluate the
    fixture tree directly on the inputs and compare bit for bit.  Inputs span a wide
    dynamic range so that a different association order changes the bits."""
    kind, P, S, p, tree = row
    rng = np.random.default_rng(100 + P * 10 + S)
    n = 3 * P + 2
    xs = [(rng.standard_normal(n) * np.exp2(rng.integers(-20, 21, n))).astype(np.float32)
          for _ in range(P)]
    run = G.simulate(P, n, S, inputs=xs, op="sum", dtype="f32")
    bounds = _mpi_partition(n, P)
    for x in range(P):
        for b in range(P):
            if (x - b) % P != p:
                continue
            lo, hi = bounds[b]
            got = run.outputs[x][lo:hi]
            want = G.eval_tree(tree, lambda k: xs[(b + k) % P][lo:hi], "sum")
            assert got.dtype == np.float32
            np.testing.assert_array_equal(got.view(np.uint32), want.view(np.uint32))


def test_association_is_observable():
    """P=5 BO: (0+((1+3)+(2+4))) on (1, 2^24, 1, -2^24, 1) gives 3 in float32, while
    the left-to-right sum gives 1 -- the pins above can tell trees apart."""
    vals = [1.0, 2.0 ** 24, 1.0, -(2.0 ** 24), 1.0]
    xs = [np.full(5, v, dtype=np.float32) for v in vals]
    out = G.allreduce(xs, 6, "sum", "f32")
    seq = np.float32(0)
    for v in vals:
        seq = np.float32(seq + np.float32(v))
    assert seq == np.float32(1.0)
    # rank x's block b (one element each): rotation b, so check block 0 (element 0)
    assert out[0][0] == np.float32(3.0)


# ---------------------------------------------------------------------------
# Step counts and the coverage invariant
# ---------------------------------------------------------------------------

def test_step_counts():
    for P in range(1, 131):
        L, Ss = _Ls(P)
        assert G.vector_counts(P)[-1] == 1 and len(G.vector_counts(P)) == L + 1
        for S in Ss:
            run = G.simulate(P, 0, S)
            red = [s for s in run.log if s["phase"] == "reduce"]
            dis = [s for s in run.log if s["phase"] == "distribute"]
            assert len(red) == L and len(dis) == L - run.r and len(run.log) == S
        for bad in (L - 1, 2 * L + 1):
            if bad >= 0:
                with pytest.raises(ValueError):
                    G.simulate(P, 0, bad)


@pytest.mark.parametrize("P", list(range(1, 41)) + [63, 64, 65, 96, 127, 128, 129, 130])
def test_every_output_covers_every_rank_once(P):
    """Each result block is a reduction over every process exactly once (the result
    u_{i,Sigma} of Sec. "Combination of distributed data vectors"), and every combine
    joins two disjoint sets of processes."""
    L, Ss = _Ls(P)
    for S in Ss:
        run = G.simulate(P, 0, S)
        ex = run.exprs
        for (kind, *rest) in ex.nodes:
            if kind == "pair":
                a, b = rest
                la, lb = set(ex.leaves(a)), set(ex.leaves(b))
                assert not (la & lb)
        for x in range(P):
            for b in range(P):
                pl, e = run.out_key[x][b]
                assert pl == (x - b) % P
        for key in set(k for row in run.out_key for k in row):
            offs = ex.leaves(key[1])
            assert sorted(offs) == list(range(P))


# ---------------------------------------------------------------------------
# Brute force on tiny integer inputs (the definition of Allreduce)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("P", range(1, 10))
def test_int32_bruteforce(P):
    rng = np.random.default_rng(P)
    L, Ss = _Ls(P)
    for n in sorted({0, 1, max(P - 1, 0), P, P + 1, 2 * P + 3, 20}):
        xs = [rng.integers(-1000, 1001, n).astype(np.int32) for _ in range(P)]
        for S in Ss:
            for op in G.OPS:
                out = G.allreduce(xs, S, op, "i32")
                ref = G.column_reduce_exact(xs, op, "i32")
                for x in range(P):
                    np.testing.assert_array_equal(out[x], ref)


def test_int32_wraparound():
    P = 7
    xs = [np.full(9, 2 ** 31 - 1 - k, dtype=np.int32) for k in range(P)]
    ref = G.column_reduce_exact(xs, "sum", "i32")
    assert ref[0] == np.int32(((7 * (2 ** 31 - 1) - 21 + 2 ** 31) % 2 ** 32) - 2 ** 31)
    for S in range(3, 7):
        for o in G.allreduce(xs, S, "sum", "i32"):
            np.testing.assert_array_equal(o, ref)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_float_max_min_exact(dtype):
    rng = np.random.default_rng(7)
    for P in (2, 5, 6, 8, 11):
        L, Ss = _Ls(P)
        n = 4 * P + 1
        xs = [rng.standard_normal(n).astype(np.float32) for _ in range(P)]
        if dtype == "bf16":
            xs = [G.round_to_bf16(v) for v in xs]
        for S in Ss:
            for op in ("max", "min"):
                out = G.allreduce(xs, S, op, dtype)
                ref = G.column_reduce_exact(xs, op, dtype)
                for o in out:
                    np.testing.assert_array_equal(o, ref)


# ---------------------------------------------------------------------------
# Traffic and computation: the paper's closed forms
# ---------------------------------------------------------------------------

def test_bandwidth_optimal_traffic():
    """eq. bo_cost: 2(P-1) blocks per process; with P | n that is 2(P-1)/P * n."""
    for P in range(2, 131):
        L = G.ceil_log2(P)
        run = G.simulate(P, 3 * P, 2 * L)
        for x in range(P):
            assert run.message_blocks_per_rank(x) == 2 * (P - 1)
            assert run.message_elems_per_rank(x) == 2 * (P - 1) * 3


def test_latency_optimal_traffic():
    """eq. lo_cost: P * ceil(log P) blocks per process."""
    for P in range(2, 131):
        L = G.ceil_log2(P)
        run = G.simulate(P, 0, L)
        for x in range(P):
            assert run.message_blocks_per_rank(x) == P * L


@pytest.mark.parametrize("P", [2, 4, 8, 16, 32, 64, 128])
def test_intermediate_traffic_power_of_two(P):
    """eq. intemediate_cost: 2(P-1) + (2^r - 1)(ceil(log P) - 1) blocks per process when
    the result count K = 2^r, i.e. P a power of two."""
    L = G.ceil_log2(P)
    for r in range(0, L):
        run = G.simulate(P, 0, 2 * L - r)
        assert run.K == 2 ** r
        assert run.message_blocks_per_rank(0) == 2 * (P - 1) + (2 ** r - 1) * (L - 1)


def test_recursive_halving_doubling_volumes():
    """Power-of-two P: BO moves Recursive Halving's 2(P-1)/P * n per process in 2 log P
    steps; LO moves Recursive Doubling's log P * n in log P steps (Secs.
    "Bandwidth-optimal algorithm" and "Moving towards latency-optimal version")."""
    for P in (2, 4, 8, 16):
        L = G.ceil_log2(P)
        n = 5 * P
        bo = G.simulate(P, n, 2 * L)
        lo = G.simulate(P, n, L)
        assert len(bo.log) == 2 * L and len(lo.log) == L
        assert bo.message_elems_per_rank(0) == 2 * (P - 1) * n // P
        assert lo.message_elems_per_rank(0) == L * n


def test_computation_counts():
    """Combines per process: BO (P-1) blocks (eq. bo_cost); intermediate at most
    (P-1) + (2^r-1)(2 ceil(log P) - 2) (eq. intemediate_cost, stated as a worst case);
    LO at most P(2 ceil(log P) - 2) (eq. lo_cost), reached at P = 127."""
    for P in range(2, 131):
        L, Ss = _Ls(P)
        for S in Ss:
            run = G.simulate(P, 0, S)
            ncomb = sum(len(c) for c in run.combines)
            r = run.r
            if r == 0:
                assert ncomb == P - 1
            elif r < L:
                assert ncomb <= (P - 1) + (2 ** r - 1) * (2 * L - 2)
            else:
                assert ncomb <= P * (2 * L - 2) or L == 1
    run = G.simulate(127, 0, 7)
    assert sum(len(c) for c in run.combines) == 127 * 12


def test_tx_sets_and_partners():
    """Per-step transmit sets and partners: eq. bo_tx_dist (indices ceil(N/2)..N-1 move),
    eq. bo_dir_perms (to x - floor(N/2)); the one extra vector t^{N_i} q'_{N_i} of the
    once-shifted schedule; all P q' vectors every step in the latency-optimal version
    (eq. for Q''_TX); distribution senders [N mod 2, ceil(N/2)-1] moved by +floor(N/2)."""
    for P in range(2, 70):
        L, Ss = _Ls(P)
        Ns = G.vector_counts(P)
        bo = G.simulate(P, 0, 2 * L)
        for st in bo.log:
            N, d = st["N"], st["d"]
            c = N - d
            assert d == N // 2
            pls = sorted(k[0] for k in st["tx"])
            if st["phase"] == "reduce":
                assert pls == list(range(c, N))
                for (src, dst, _items) in st["messages"]:
                    assert dst == (src - d) % P
            else:
                assert pls == list(range(N % 2, c))
                for (src, dst, _items) in st["messages"]:
                    assert dst == (src + d) % P
        if L >= 2:
            one = G.simulate(P, 0, 2 * L - 1)     # K = N_{L-1} = 2
            assert one.K == 2
            for st in one.log:
                if st["phase"] != "reduce":
                    continue
                N = st["N"]
                c = N - N // 2
                want = sorted(set(list(range(c, N)) + [N % P]))
                assert sorted(k[0] for k in st["tx"]) == want
        lo = G.simulate(P, 0, L)
        for st in lo.log:
            assert sorted(k[0] for k in st["tx"]) == list(range(P))
            assert all(not lo.exprs.is_leaf(k[1]) or st["i"] == 0 for k in st["tx"])


def test_p7_first_step_state():
    """The P=7 instance of eq. bo_step_odd: Q_1 = t^0 q_0 : t^1 (q_1+q_4) :
    t^2 (q_2+q_5) : t^3 (q_3+q_6)."""
    run = G.simulate(7, 0, 6)
    st = [(pl, run.exprs.tree(e)) for (pl, e) in run.states[0][0]]
    assert st == [(0, 0), (1, (1, 4)), (2, (2, 5)), (3, (3, 6))]


def test_latency_optimal_keeps_q_star_apart():
    """Sec. "Latency-optimal version": after an odd step every placement carries both a
    q* and a q' vector (2P vectors), which are never combined with each other."""
    for P in (3, 5, 7, 9, 127):
        L = G.ceil_log2(P)
        run = G.simulate(P, 0, L)
        keys = set(k for q in run.states[0] for k in q)
        # after step 0 (odd N): q*_k = leaf k and q'_k = (k + (k+d)) for every k
        assert len(keys) == 2 * P
        for (pl, e) in keys:
            leaves = run.exprs.leaves(e)
            assert leaves[0] == pl


# ---------------------------------------------------------------------------
# Rank agreement and rotations
# ---------------------------------------------------------------------------

def test_bo_all_ranks_identical_and_lo_rotated():
    rng = np.random.default_rng(11)
    gold = {(k, P, S, p): t for (k, P, S, p, t) in _golden()}
    for P in (5, 7):
        L = G.ceil_log2(P)
        n = 2 * P + 3
        xs = [(rng.standard_normal(n) * np.exp2(rng.integers(-12, 13, n))).astype(np.float32)
              for _ in range(P)]
        bo = G.allreduce(xs, 2 * L, "sum", "f32")
        for x in range(1, P):
            np.testing.assert_array_equal(bo[x].view(np.uint32), bo[0].view(np.uint32))
    # LO P=5: rank x's result is the P=5 tree with leaf k read from rank x+k
    T = gold[("bo", 5, 6, 0)]
    P, n = 5, 13
    xs = [(rng.standard_normal(n) * np.exp2(rng.integers(-12, 13, n))).astype(np.float32)
          for _ in range(P)]
    lo = G.allreduce(xs, 3, "sum", "f32")
    for x in range(P):
        want = G.eval_tree(T, lambda k: xs[(x + k) % P], "sum")
        np.testing.assert_array_equal(lo[x].view(np.uint32), want.view(np.uint32))


# ---------------------------------------------------------------------------
# Block partition (eq. initial_data with u = m/P, Sec. "Communication model";
# reading C3 for P not dividing n)
# ---------------------------------------------------------------------------

# (n, P, block sizes in order), written out by hand from reading C3: the first n mod P
# blocks get one element more than floor(n / P); n < P leaves the last blocks empty.
BLOCK_SIZES = [
    (1024, 5, [205, 205, 205, 205, 204]),
    (16_777_216, 24, [699_051] * 16 + [699_050] * 8),
    (4_194_304, 127, [33_027] * 2 + [33_026] * 125),
    (262_144, 8, [32_768] * 8),
    (3, 5, [1, 1, 1, 0, 0]),
    (0, 4, [0, 0, 0, 0]),
    (7, 1, [7]),
    (106, 6, [18, 18, 18, 18, 17, 17]),
    (106, 7, [16] * 1 + [15] * 6),
]


@pytest.mark.parametrize("n,P,sizes", BLOCK_SIZES, ids=lambda v: str(v) if not isinstance(v, list) else "")
def test_block_bounds_reading_c3(n, P, sizes):
    """Block i is [sum of sizes before i, + sizes[i]): contiguous, in block order, from 0
    to n, with the sizes written out above."""
    assert sum(sizes) == n and len(sizes) == P
    bounds = G.block_bounds(n, P)
    assert len(bounds) == P
    start = 0
    for (lo, hi), size in zip(bounds, sizes):
        assert (lo, hi) == (start, start + size)
        start += size
    assert start == n


def _block_pins_pass() -> bool:
    try:
        for n, P, sizes in BLOCK_SIZES:
            test_block_bounds_reading_c3(n, P, sizes)
    except AssertionError:
        return False
    return True


def _remainder_last(n, P):
    q, rem = divmod(n, P)
    out, start = [], 0
    for i in range(P):
        size = q + (1 if i >= P - rem else 0)
        out.append((start, start + size))
        start += size
    return out


def _remainder_in_last_block(n, P):
    q, rem = divmod(n, P)
    out = [(i * q, (i + 1) * q) for i in range(P)]
    out[-1] = (out[-1][0], n)
    return out


@pytest.mark.parametrize("bad", [_remainder_last, _remainder_in_last_block])
def test_planted_partition_mistake_is_caught(monkeypatch, bad):
    """Two plausible misreadings of reading C3 -- the longer blocks at the end, or the
    whole remainder in block P-1 -- fail the hand-written sizes, and they also change
    the simulation's results against checkers that partition on their own (the golden
    tree values and the textbook Ring below).  (Recursive Halving cannot see it: its
    tree is the same butterfly for every block.)"""
    monkeypatch.setattr(G, "block_bounds", bad)
    assert not _block_pins_pass()
    row = next(r for r in _golden() if r[1] == 7)
    with pytest.raises(AssertionError):
        test_golden_tree_values(row)
    with pytest.raises(AssertionError):
        test_ring_equals_textbook_ring(5)


def test_tree_notation_round_trip():
    """The fixture notation of tests/golden: hand-written strings and their trees."""
    cases = {"3": 3, "(0+1)": (0, 1), "((0+1)+(2+(3+4)))": ((0, 1), (2, (3, 4))),
             "(12+(0+7))": (12, (0, 7))}
    for text, tree in cases.items():
        assert G.parse_tree(text) == tree
        assert G.tree_string(tree) == text


def test_is_bf16_exact():
    assert G.is_bf16_exact(np.float32([0.0, 1.0, -2.5, 2.0 ** 127, 2.0 ** -120, -1.5 * 2.0 ** 60]))
    for v in (1.0 + 2.0 ** -8, 1.0 + 2.0 ** -23, 0.1):
        assert not G.is_bf16_exact(np.float32([1.0, v]))


def test_column_reduce_exact_brute_force():
    """The definition, checked against pure-Python loops over tiny inputs: int32 sums
    wrap modulo 2^32 (two's complement), max and min pick the extreme value."""
    rng = np.random.default_rng(21)
    for P in (1, 2, 5, 9):
        xs = [rng.integers(-2**31, 2**31, 13, dtype=np.int64).astype(np.int32) for _ in range(P)]
        for op in ("sum", "max", "min"):
            got = G.column_reduce_exact(xs, op, "i32")
            for e in range(13):
                col = [int(x[e]) for x in xs]
                if op == "sum":
                    t = sum(col) & 0xFFFFFFFF
                    want = t - 2**32 if t >= 2**31 else t
                else:
                    want = max(col) if op == "max" else min(col)
                assert int(got[e]) == want
        fs = [rng.standard_normal(13).astype(np.float32) for _ in range(P)]
        for op in ("max", "min"):
            got = G.column_reduce_exact(fs, op, "f32")
            for e in range(13):
                col = [float(x[e]) for x in fs]
                assert float(got[e]) == (max(col) if op == "max" else min(col))


# ---------------------------------------------------------------------------
# The compensated reference sum (the Kahan reference of the float tolerance)
# ---------------------------------------------------------------------------

def _kahan_cases():
    rng = np.random.default_rng(11)
    cases = []
    for P in (2, 5, 24, 127):
        x = rng.standard_normal((P, 500)) * np.exp2(rng.integers(-30, 31, (P, 500)))
        cases.append(x)
    # heavy cancellation: large terms of both signs around small ones
    big = rng.standard_normal((40, 300)) * 1e12
    cases.append(np.concatenate([big, rng.standard_normal((40, 300)), -big[::-1]]))
    return cases


def test_kahan_sum_within_compensated_bound():
    """Compensated summation of P terms has |error| <= (2u + O(P u^2)) sum|x| with
    u = 2^-53 (the standard bound for Kahan's method); the exact sum comes from
    math.fsum, which rounds the exact sum once.  A plain float64 sum of these inputs
    does not meet the bound, so a broken compensation fails it."""
    import math
    u = 2.0 ** -53
    for x in _kahan_cases():
        P = x.shape[0]
        s, mag = G.kahan_sum_f64(list(x))
        exact = np.array([math.fsum(x[:, j]) for j in range(x.shape[1])])
        want_mag = np.array([math.fsum(np.abs(x[:, j])) for j in range(x.shape[1])])
        np.testing.assert_allclose(mag, want_mag, rtol=P * u, atol=0)
        assert np.all(np.abs(s - exact) <= (2 * u + 2 * P * u * u) * want_mag)


def test_kahan_sum_recovers_lost_low_bits():
    """1 + 1000 * 2^-60: every addend is below half an ulp of 1, so rank-order plain
    summation returns exactly 1.0, while compensated summation returns the correctly
    rounded 1 + 1000 * 2^-60 (= 1 + 4 * 2^-52)."""
    import math
    col = [1.0] + [2.0 ** -60] * 1000
    s, _ = G.kahan_sum_f64([np.array([v]) for v in col])
    assert s[0] == math.fsum(col) == 1.0 + 4 * 2.0 ** -52


def test_planted_kahan_sign_flip_is_caught(monkeypatch):
    """The compensation term with its sign flipped (c = y - (t - s)) fails both pins."""
    def flipped(inputs):
        stack = np.stack([np.asarray(v, dtype=np.float64) for v in inputs])
        s = np.zeros(stack.shape[1])
        comp = np.zeros_like(s)
        for row in stack:
            y = row - comp
            t = s + y
            comp = y - (t - s)
            s = t
        return s, np.abs(stack).sum(axis=0)
    monkeypatch.setattr(G, "kahan_sum_f64", flipped)
    with pytest.raises(AssertionError):
        test_kahan_sum_within_compensated_bound()
    with pytest.raises(AssertionError):
        test_kahan_sum_recovers_lost_low_bits()


# ---------------------------------------------------------------------------
# Floating point: error bounds and bf16
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("P", [2, 3, 5, 8, 13, 24, 33])
def test_f32_within_tree_error_bound(P):
    """A summation tree of height h has |error| <= h * 2^-24 * sum|x| (to first order).
    Each reduction step adds at most one level, so h <= L = ceil(log2 P)."""
    rng = np.random.default_rng(P)
    L, Ss = _Ls(P)
    n = 7 * P + 5
    xs = [rng.uniform(-1, 1, n).astype(np.float32) for _ in range(P)]
    ref, mag = G.kahan_sum_f64(xs)
    for S in Ss:
        run = G.simulate(P, n, S, inputs=xs)
        height = max(_height(run.exprs.tree(k[1])) for row in run.out_key for k in row)
        assert height <= L
        for o in run.outputs:
            err = np.abs(o.astype(np.float64) - ref)
            assert np.all(err <= height * 2.0 ** -24 * mag * (1 + 1e-6) + 1e-30)


def _height(t):
    if isinstance(t, int):
        return 0
    return 1 + max(_height(t[0]), _height(t[1]))


def test_bf16_rounding_matches_library():
    rng = np.random.default_rng(3)
    x = np.concatenate([
        rng.standard_normal(100000).astype(np.float32),
        (rng.standard_normal(1000) * 1e30).astype(np.float32),
        (rng.standard_normal(1000) * 1e-30).astype(np.float32),
        # exact ties: low half == 0x8000, with odd and even upper halves
        (np.arange(1000, dtype=np.uint32) << 16 | np.uint32(0x8000)).view(np.float32),
        np.array([0.0, 1.0, -1.0, 65504.0], dtype=np.float32),
    ])
    x = x[np.isfinite(x)]
    mine = G.round_to_bf16(x)
    lib = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    np.testing.assert_array_equal(mine.view(np.uint32), lib.view(np.uint32))


def test_bf16_sum_rounds_once():
    """bf16 inputs, float32 accumulation, one final rounding: the result is a bf16 value
    within 2^-8 relative of the float32 tree result, which itself is within the tree
    bound of the exact sum."""
    rng = np.random.default_rng(5)
    P, n = 7, 40
    xs = [G.round_to_bf16(rng.standard_normal(n).astype(np.float32)) for _ in range(P)]
    ref, mag = G.kahan_sum_f64(xs)
    for S in range(3, 7):
        for o in G.allreduce(xs, S, "sum", "bf16"):
            assert G.is_bf16_exact(o)
            err = np.abs(o.astype(np.float64) - ref)
            assert np.all(err <= 2.0 ** -8 * np.abs(ref) + 3 * 2.0 ** -24 * mag + 1e-30)


# ---------------------------------------------------------------------------
# Degenerate cases and element subsets
# ---------------------------------------------------------------------------

def test_degenerate_cases():
    x = [np.arange(5, dtype=np.float32)]
    out = G.allreduce(x, 0, "sum", "f32")
    np.testing.assert_array_equal(out[0], x[0])           # P = 1: no-op
    ys = [np.ones(0, np.float32) for _ in range(4)]
    assert all(len(o) == 0 for o in G.allreduce(ys, 3, "sum", "f32"))   # n = 0
    a = np.float32([1.5, -2.0, 3.25])
    b = np.float32([0.25, 8.0, -1.0])
    for S in (1, 2):                                          # P = 2
        for o in G.allreduce([a, b], S, "sum", "f32"):
            np.testing.assert_array_equal(o, a + b)


def test_element_subset_matches_full_run():
    rng = np.random.default_rng(9)
    P, n = 7, 101
    xs = [rng.standard_normal(n).astype(np.float32) for _ in range(P)]
    sel = np.sort(rng.choice(n, 23, replace=False))
    for S in range(3, 7):
        full = G.allreduce(xs, S, "sum", "f32")
        part = G.allreduce(xs, S, "sum", "f32", elements=sel)
        for x in range(P):
            np.testing.assert_array_equal(part[x], full[x][sel])


def test_cost_model_argmin_matches_paper_example():
    """Eq. opt_number_of_steps with Table 2's parameters for P=127, m=9 KiB gives
    r = log2(alpha / (m (beta + 2 gamma))) + log2(P / ((log2 P - 1) ln 2)) ~ 3.3, i.e.
    S ~ 14 - 3 = 11; the integer argmin of eq. intemediate_cost agrees."""
    import math
    a, b, g = 3e-5, 1e-8, 2e-10
    P, m = 127, 9 * 1024
    r = math.log2(a / (m * (b + 2 * g))) + math.log2(P / ((math.log2(P) - 1) * math.log(2)))
    assert 3.0 < r < 3.5
    assert G.optimal_steps(P, m, a, b, g) == 14 - round(r)


# ---------------------------------------------------------------------------
# Planted mistakes: each must make at least one pin fail
# ---------------------------------------------------------------------------

def _pins_pass() -> bool:
    try:
        for row in _golden():
            test_golden_tree(row)
        for P in (3, 5, 6, 7):
            test_int32_bruteforce(P)
        test_bandwidth_optimal_traffic()
    except (AssertionError, KeyError, ValueError, IndexError):
        return False
    return True


def test_pins_pass_unmodified():
    assert _pins_pass()


def test_planted_wrong_partner_is_caught(monkeypatch):
    monkeypatch.setattr(G, "_reduce_partner", lambda x, d, P, group="cyclic": (x + d) % P)
    assert not _pins_pass()


def test_planted_sign_error_is_caught(monkeypatch):
    real = G._combine
    monkeypatch.setattr(G, "_combine", lambda op, a, b: a - b if op == "sum" else real(op, a, b))
    assert not _pins_pass()


def test_planted_floor_halving_is_caught(monkeypatch):
    def bad_counts(P):
        Ns = [P]
        while Ns[-1] > 1:
            Ns.append(max(1, Ns[-1] // 2))
        return Ns
    monkeypatch.setattr(G, "vector_counts", bad_counts)
    assert not _pins_pass()


# ---------------------------------------------------------------------------
# The self-inverse group of Table 1b (XOR group, P a power of two)
# ---------------------------------------------------------------------------

POW2 = [2, 4, 8, 16, 32, 64]


def _textbook_recursive_halving(xs):
    """Reduce-scatter by recursive vector halving, then allgather by recursive doubling,
    with the partner at distance P/2 first (each rank keeps the half of its blocks whose
    index agrees with its own rank in the exchanged bit).  Written from the textbook
    description, independently of the oracle's schedule simulation."""
    P, n = len(xs), len(xs[0])
    bounds = _mpi_partition(n, P)
    buf = [x.copy() for x in xs]
    resp = [list(range(P)) for _ in range(P)]
    m = P // 2
    while m >= 1:
        new = [b.copy() for b in buf]
        new_resp = []
        for x in range(P):
            y = x ^ m
            keep = [b for b in resp[x] if (b & m) == (x & m)]
            for b in keep:
                lo, hi = bounds[b]
                new[x][lo:hi] = buf[x][lo:hi] + buf[y][lo:hi]
            new_resp.append(keep)
        buf, resp = new, new_resp
        m //= 2
    m = 1
    while m < P:
        new = [b.copy() for b in buf]
        new_resp = []
        for x in range(P):
            y = x ^ m
            for b in resp[y]:
                lo, hi = bounds[b]
                new[x][lo:hi] = buf[y][lo:hi]
            new_resp.append(resp[x] + resp[y])
        buf, resp = new, new_resp
        m *= 2
    return buf


def _textbook_recursive_doubling(xs):
    """Every rank exchanges its whole vector with the partner at distance P/2, P/4, ...,
    1 and adds the partner's vector to its own."""
    P = len(xs)
    v = [x.copy() for x in xs]
    m = P // 2
    while m >= 1:
        v = [v[x] + v[x ^ m] for x in range(P)]
        m //= 2
    return v


@pytest.mark.parametrize("P", POW2)
def test_xor_group_bo_is_recursive_halving(P):
    """Sec. "Bandwidth-optimal algorithm": with P a power of two and the group of Table
    1b the bandwidth-optimal algorithm is Recursive Halving -- same bits in float32."""
    rng = np.random.default_rng(P)
    n = 5 * P + 3
    xs = [(rng.standard_normal(n) * np.exp2(rng.integers(-20, 21, n))).astype(np.float32)
          for _ in range(P)]
    L = G.ceil_log2(P)
    got = G.allreduce(xs, 2 * L, "sum", "f32", group="xor")
    want = _textbook_recursive_halving(xs)
    for x in range(P):
        np.testing.assert_array_equal(got[x].view(np.uint32), want[x].view(np.uint32))


@pytest.mark.parametrize("P", POW2)
def test_xor_group_lo_is_recursive_doubling(P):
    """Sec. "Moving towards latency-optimal version": with the group of Table 1b the
    latency-optimal algorithm is Recursive Doubling -- same bits in float32."""
    rng = np.random.default_rng(100 + P)
    n = 3 * P + 1
    xs = [(rng.standard_normal(n) * np.exp2(rng.integers(-20, 21, n))).astype(np.float32)
          for _ in range(P)]
    got = G.allreduce(xs, G.ceil_log2(P), "sum", "f32", group="xor")
    want = _textbook_recursive_doubling(xs)
    for x in range(P):
        np.testing.assert_array_equal(got[x].view(np.uint32), want[x].view(np.uint32))


@pytest.mark.parametrize("P", POW2)
def test_xor_group_coverage_bruteforce_and_traffic(P):
    """Every result covers every rank once, int32 results are the column sums, and the
    per-rank traffic is Recursive Halving's 2(P-1) blocks (S = 2L), Recursive Doubling's
    P L blocks (S = L), and 2(P - K) + r K blocks in between (K = 2^r result copies: r
    halving steps are replaced by doubling steps on K-block vectors)."""
    L = G.ceil_log2(P)
    rng = np.random.default_rng(7 * P)
    n = 2 * P + 1
    xs = [rng.integers(-1000, 1001, n).astype(np.int32) for _ in range(P)]
    ref = G.column_reduce_exact(xs, "sum", "i32")
    for S in range(L, 2 * L + 1):
        run = G.simulate(P, n, S, inputs=xs, dtype="i32", group="xor")
        for o in run.outputs:
            np.testing.assert_array_equal(o, ref)
        for key in set(k for row in run.out_key for k in row):
            assert sorted(run.exprs.leaves(key[1])) == list(range(P))
        r, K = run.r, run.K
        assert K == 2 ** r
        for x in range(P):
            assert run.message_blocks_per_rank(x) == 2 * (P - K) + r * K
        for st in run.log:
            d = st["d"]
            for (src, dst, _items) in st["messages"]:
                assert dst == src ^ d          # pairwise exchange partners


def test_xor_group_needs_power_of_two():
    with pytest.raises(ValueError):
        G.simulate(6, 0, 4, group="xor")


# ---------------------------------------------------------------------------
# The Ring algorithm (Sec. "Allreduce as permutation composition", cyclic case)
# ---------------------------------------------------------------------------

def _textbook_ring(xs):
    """Ring Allreduce as usually described: P-1 reduce-scatter steps in which rank x
    passes its running partial of chunk (x - i) mod P to rank x + 1, which adds its own
    chunk to it, then P-1 allgather steps passing the finished chunks on.  Written
    independently of the oracle's schedule simulation."""
    P, n = len(xs), len(xs[0])
    bounds = _mpi_partition(n, P)
    buf = [x.copy() for x in xs]
    for i in range(P - 1):
        new = [b.copy() for b in buf]
        for x in range(P):
            c = (x - i) % P
            y = (x + 1) % P
            lo, hi = bounds[c]
            new[y][lo:hi] = buf[y][lo:hi] + buf[x][lo:hi]
        buf = new
    for i in range(P - 1):
        new = [b.copy() for b in buf]
        for x in range(P):
            c = (x + 1 - i) % P
            y = (x + 1) % P
            lo, hi = bounds[c]
            new[y][lo:hi] = buf[x][lo:hi]
        buf = new
    return buf


@pytest.mark.parametrize("P", [2, 3, 5, 7, 8, 13, 24])
def test_ring_equals_textbook_ring(P):
    rng = np.random.default_rng(200 + P)
    n = 3 * P + 2
    xs = [(rng.standard_normal(n) * np.exp2(rng.integers(-20, 21, n))).astype(np.float32)
          for _ in range(P)]
    got = G.allreduce(xs, "ring", "sum", "f32")
    want = _textbook_ring(xs)
    for x in range(P):
        np.testing.assert_array_equal(got[x].view(np.uint32), want[x].view(np.uint32))


@pytest.mark.parametrize("P", [1, 2, 3, 4, 5, 9, 16, 31])
def test_ring_steps_traffic_and_tree(P):
    """2(P-1) steps, 2(P-1) blocks and P-1 combines per rank (eq. naive_cost); the
    result is the chain of eq. ring_reduce: q_{P-1} (+) (... (+) (q_1 (+) q_0))."""
    rng = np.random.default_rng(P)
    n = 2 * P + 1
    xs = [rng.integers(-1000, 1001, n).astype(np.int32) for _ in range(P)]
    run = G.simulate_ring(P, n, inputs=xs, dtype="i32")
    assert len(run.log) == 2 * (P - 1)
    ref = G.column_reduce_exact(xs, "sum", "i32")
    for o in run.outputs:
        np.testing.assert_array_equal(o, ref)
    for x in range(P):
        assert run.message_blocks_per_rank(x) == 2 * (P - 1)
    assert sum(len(c) for c in run.combines) == P - 1
    if P >= 2:
        chain = 0
        for k in range(1, P):
            chain = (k, chain)
        assert run.exprs.tree(run.after_reduction[0][1]) == chain


# ---------------------------------------------------------------------------
# Step counts beyond 2L: fold schedules toward the Ring (reading C19)
# ---------------------------------------------------------------------------

def _fold_cases():
    out = []
    for P in list(range(3, 41)) + [64, 127]:
        L = G.ceil_log2(P)
        Ss = list(range(2 * L + 2, 2 * (P - 1) + 1, 2))
        if P > 40:
            Ss = Ss[:3] + Ss[-2:]
        out += [(P, S) for S in Ss]
    return out


@pytest.mark.parametrize("P,S", _fold_cases())
def test_fold_schedule(P, S):
    """Every even step count from 2L to 2(P-1): S steps; bandwidth-optimal traffic of
    2(P-1) blocks per rank (eq. bo_cost's volume) whatever S; step i moves f_i <=
    floor(N_i/2) blocks to rank x - f_i; every result covers every rank once; int32
    results are the column sums; all ranks hold identical bits (one result copy)."""
    L = G.ceil_log2(P)
    F = S // 2
    folds = G.fold_sequence(P, F)
    assert len(folds) == F and sum(folds) == P - 1
    N = P
    for f in folds:
        assert 1 <= f <= N // 2
        N -= f
    rng = np.random.default_rng(P * 100 + S)
    n = 2 * P + 3
    xs = [rng.integers(-1000, 1001, n).astype(np.int32) for _ in range(P)]
    run = G.simulate(P, n, S, inputs=xs, dtype="i32")
    assert len(run.log) == S and run.K == 1
    ref = G.column_reduce_exact(xs, "sum", "i32")
    for o in run.outputs:
        np.testing.assert_array_equal(o, ref)
    for x in range(P):
        assert run.message_blocks_per_rank(x) == 2 * (P - 1)
    red = [st for st in run.log if st["phase"] == "reduce"]
    for st, f in zip(red, folds):
        assert len(st["tx"]) == f
        for (src, dst, _items) in st["messages"]:
            assert dst == (src - f) % P
    key = run.after_reduction[0]
    assert sorted(run.exprs.leaves(key[1])) == list(range(P))
    fx = [(rng.standard_normal(n) * np.exp2(rng.integers(-12, 13, n))).astype(np.float32)
          for _ in range(P)]
    outs = G.allreduce(fx, S, "sum", "f32")
    for x in range(1, P):
        np.testing.assert_array_equal(outs[x].view(np.uint32), outs[0].view(np.uint32))


def test_fold_schedule_ends():
    """F = L folds are the bandwidth-optimal halving; S = 2(P-1) folds one vector per step
    and reduces to the chain q_0 (+) (q_1 (+) (... (+) (q_{P-2} (+) q_{P-1})))."""
    for P in (5, 8, 13):
        L = G.ceil_log2(P)
        assert G.fold_sequence(P, L) == [N // 2 for N in G.vector_counts(P)[:-1]]
        run = G.simulate(P, 0, 2 * (P - 1))
        chain = P - 1
        for k in range(P - 2, -1, -1):
            chain = (k, chain)
        assert run.exprs.tree(run.after_reduction[0][1]) == chain
    with pytest.raises(ValueError):
        G.simulate(8, 0, 9)                      # odd S beyond 2L
    with pytest.raises(ValueError):
        G.simulate(8, 0, 16)                     # beyond 2(P-1)


# ---------------------------------------------------------------------------
# A second implementation of the definition (oracle/column_reduce.c)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("threads", [1, 3])
def test_column_reduce_is_the_definition(threads):
    """The C column reduction against numpy's column reduction: int32 wraparound sums
    and max/min exactly, fp32 sums within the rank-order rounding of a float64 sum."""
    from oracle import column_reduce as CR
    rng = np.random.default_rng(11)
    P, n = 7, 1001
    xi = [rng.integers(-2 ** 31, 2 ** 31, n, dtype=np.int64).astype(np.int32) for _ in range(P)]
    want = np.zeros(n, np.int64)
    for v in xi:
        want += v
    want = ((want + 2 ** 31) % 2 ** 32 - 2 ** 31).astype(np.int32)
    for o in CR.column_allreduce(xi, "sum", "i32", threads):
        np.testing.assert_array_equal(o, want)
    for op, f in (("max", np.max), ("min", np.min)):
        for dt, xs in (("i32", xi), ("f32", [v.astype(np.float32) for v in xi])):
            for o in CR.column_allreduce(xs, op, dt, threads):
                np.testing.assert_array_equal(o, f(np.stack(xs), axis=0))
    xf = [rng.standard_normal(n).astype(np.float32) for _ in range(P)]
    exact = np.sum(np.stack(xf).astype(np.float64), axis=0)
    for o in CR.column_allreduce(xf, "sum", "f32", threads):
        np.testing.assert_array_equal(o, exact.astype(np.float32))


@pytest.mark.parametrize("P", [2, 3, 5, 7, 8, 12, 24, 33])
def test_oracle_order_free_results_equal_column_reduce(P):
    """Where the result does not depend on the association order (int32 wraparound sum,
    max, min), every schedule of the oracle -- every S, both groups, folds, the Ring --
    equals the plain column reduction bit for bit."""
    from oracle import column_reduce as CR
    rng = np.random.default_rng(100 + P)
    n = 3 * P + 2
    xi = [rng.integers(-2 ** 31, 2 ** 31, n, dtype=np.int64).astype(np.int32) for _ in range(P)]
    xf = [rng.standard_normal(n).astype(np.float32) for _ in range(P)]
    L = G.ceil_log2(P)
    sched = [(S, "cyclic") for S in range(L, 2 * L + 1)]
    sched += [(S, "cyclic") for S in range(2 * L + 2, 2 * (P - 1) + 1, 2)]
    if P & (P - 1) == 0:
        sched += [(S, "xor") for S in range(L, 2 * L + 1)]
    for (S, group) in sched + [("ring", "cyclic")]:
        for (dt, xs, op) in (("i32", xi, "sum"), ("i32", xi, "max"), ("f32", xf, "min")):
            want = CR.column_allreduce(xs, op, dt)[0]
            for o in G.allreduce(xs, S, op, dt, group=group):
                np.testing.assert_array_equal(o, want, err_msg=f"P={P} S={S} {group} {dt} {op}")


@pytest.mark.parametrize("P", [3, 5, 8, 24, 33, 127])
def test_cost_model_beyond_2L_joins_the_paper_equations(P):
    """Fold schedules cost S alpha plus the bandwidth-optimal traffic and combines: the
    first fold (S = 2L + 2) is eq. bo_cost plus exactly two alpha terms, the last
    (S = 2(P - 1)) is eq. naive_cost, the Ring's, and the traffic terms of every fold
    are those the oracle's fold simulation sends (2(P - 1) blocks per rank)."""
    L = G.ceil_log2(P)
    m = 9.0 * 1024 * P
    for (a, b, c) in [(1e-5, 1e-9, 1e-10), (2.5e-6, 0.0, 3e-13), (0.0, 1e-9, 0.0)]:
        ring = G.cost_model_time(P, m, "ring", a, b, c)
        if 2 * (P - 1) > 2 * L:
            first = G.cost_model_time(P, m, 2 * L + 2, a, b, c)
            assert first == pytest.approx(G.cost_model_time(P, m, 2 * L, a, b, c) + 2 * a, rel=1e-12, abs=1e-300)
            assert G.cost_model_time(P, m, 2 * (P - 1), a, b, c) == pytest.approx(ring, rel=1e-12, abs=1e-300)
    n = 7 * P
    for S in range(2 * L + 2, 2 * (P - 1) + 1, 2):
        run = G.simulate(P, n, S)
        # all ranks together send 2(P - 1) n 4 bytes; the beta-only model per rank,
        # 2(P - 1) u with u = m / P and m = 4 n, is that total over P
        assert sum(run.step_bytes()) == 2 * (P - 1) * n * 4
        assert G.cost_model_time(P, n * 4.0, S, 0.0, 1.0, 0.0) == pytest.approx(sum(run.step_bytes()) / P)

