"""Host-side checks of libgar's schedule builder against the CPU oracle (no GPU).

* the library loads and exports every function include/gar.h declares;
* per communication step: transmitted placements, partner offset and message bytes
  equal the oracle's simulated messages;
* the origin map and the fused program's result trees equal the oracle's;
* the step-faithful op tables, executed on the CPU with the kernels' semantics (all
  reads of a launch see the state before it), give the oracle's results bit for bit
  and never write a block another op of the same launch reads;
* argument errors return the documented codes.
"""

import os
import re

import numpy as np
import pytest
import torch

from oracle import gar_oracle as G
from paper_2004_09362_gb300 import gar

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
BUF_NONE, BUF_RANK, BUF_QP0, BUF_QP1, BUF_QS = range(5)


def test_library_exports_every_declared_function():
    with open(os.path.join(ROOT, "include", "gar.h")) as f:
        hdr = f.read()
    declared = set(re.findall(r"GAR_API\s+[\w\s\*]*?\b(gar_\w+)\s*\(", hdr))
    assert declared, "no declarations found"
    assert declared == set(gar.EXPORTS)
    import ctypes
    lib = ctypes.CDLL(gar.lib_path())
    for name in declared:
        assert hasattr(lib, name), name
        # the binding has a wrapper of the same name for every entry point
        assert callable(getattr(gar, name, None)), name
    # the binding's copies of the header's limits
    for name in ("GAR_MAX_P", "GAR_FUSED_MAX_OPS"):
        m = re.search(r"#define\s+" + name + r"\s+(\d+)", hdr)
        assert m and int(m.group(1)) == getattr(gar, name), name


def test_jit_compiles_without_gpu():
    gar.gar_selftest_compile()


def _cases():
    out = []
    for P in list(range(1, 41)) + [63, 64, 65, 127, 128, 129]:
        L = G.ceil_log2(P)
        for S in range(L, 2 * L + 1):
            out.append((P, S, "cyclic"))
    for P in (1, 2, 4, 8, 16, 32, 64, 128):
        L = G.ceil_log2(P)
        for S in range(L, 2 * L + 1):
            out.append((P, S, "xor"))
    for P in list(range(4, 34)) + [64, 127]:      # fold schedules: even S in (2L, 2(P-1)]
        L = G.ceil_log2(P)
        for S in range(2 * L + 2, 2 * (P - 1) + 1, 2):
            out.append((P, S, "cyclic"))
    return out


@pytest.mark.parametrize("P,S,group", _cases())
def test_schedule_matches_oracle(P, S, group):
    n = 3 * P + 1 if P > 1 else 5
    for dtype in ("f32", "bf16"):
        plan = gar.gar_plan_create_group(P, n, dtype, "sum", S, group)
        info = plan.info()
        assert info["group"] == gar.GROUPS[group]
        run = G.simulate(P, n, S, dtype=dtype, group=group)
        assert (info["L"], info["S"], info["r"], info["K"]) == (run.L, run.steps, run.r, run.K)
        ws, per_step, S_lib = gar.gar_plan_bytes(plan)
        assert S_lib == S
        assert per_step == run.step_bytes()
        for t, st in enumerate(run.log):
            phase, partner, tx = gar.gar_plan_step(plan, t)
            assert phase == (0 if st["phase"] == "reduce" else 1)
            if group == "xor":
                assert partner == st["d"]
            else:
                assert partner == (st["d"] if phase == 0 else -st["d"])
            assert sorted(tx) == sorted(k[0] for k in st["tx"])
        # origin map: rank x's block b comes from placement (x - b); its tree is copy o
        origin = gar.gar_plan_origin(plan)
        root_of = {key[1]: s for s, key in enumerate(run.after_reduction)}
        for p in range(P):
            key = run.out_key[p % P][0]       # rank p, block 0 -> placement p
            assert key[0] == p
            assert root_of[key[1]] == origin[p]
        # fused program trees == the oracle's result trees
        pairs, outs = gar.gar_plan_fused_program(plan)
        memo = {}

        def tree(v):
            if v < P:
                return v
            if v not in memo:
                a, b = pairs[v - P]
                memo[v] = (tree(a), tree(b))
            return memo[v]

        assert len(outs) == run.K
        for s in range(run.K):
            assert tree(outs[s]) == run.exprs.tree(run.after_reduction[s][1])


def _blocks(n, P):
    return G.block_bounds(n, P)


def _to_acc(a, dtype):
    return a.astype(np.int32 if dtype == "i32" else np.float32)


def _round_store(a, dtype):
    if dtype == "bf16":
        return torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(torch.bfloat16).float().numpy()
    return a


def _op(op, a, b):
    if op == "sum":
        return a + b
    return np.maximum(a, b) if op == "max" else np.minimum(a, b)


def emulate_step_faithful(plan, xs, dtype, op, group="cyclic"):
    """Executes the plan's step-faithful op table on the CPU.  Rank buffers hold the
    element type (bf16 values kept as float32 after rounding), workspace the
    accumulation type.  Returns (outputs, per-launch recv element counts)."""
    P = len(xs)
    n = len(xs[0])
    bounds = _blocks(n, P)
    acc_dt = np.int32 if dtype == "i32" else np.float32
    bufs = {BUF_RANK: [x.copy() for x in xs],
            BUF_QP0: [np.zeros(n, acc_dt) for _ in range(P)],
            BUF_QP1: [np.zeros(n, acc_dt) for _ in range(P)],
            BUF_QS: [np.zeros(n, acc_dt) for _ in range(P)]}
    ops, partners = gar.gar_plan_step_ops(plan)
    xr = group == "xor"
    for l, partner in enumerate(partners):
        lops = ops[ops[:, 0] == l]
        writes, reads, written = [], set(), {}
        for (_l, recv_place, dst_place, recv_buf, o0b, o0o, o1b, o1o) in lops:
            for x in range(P):
                b = (x ^ dst_place) if xr else (x - dst_place) % P
                lo, hi = bounds[b]
                recv = None
                if recv_place >= 0:
                    src = (x ^ partner) if xr else (x + partner) % P
                    # the partner holds the same block at the transmitted placement
                    assert ((src ^ recv_place) if xr else (src - recv_place) % P) == b
                    recv = _to_acc(bufs[recv_buf][src][lo:hi], dtype)
                    reads.add((recv_buf, src, b))
                for (ob, oo) in ((o0b, o0o), (o1b, o1o)):
                    if ob == BUF_NONE:
                        continue
                    if oo != BUF_NONE:
                        own = _to_acc(bufs[oo][x][lo:hi], dtype)
                        if oo != ob:
                            reads.add((oo, x, b))
                        val = own if recv is None else _op(op, own, recv)
                    else:
                        val = recv
                    key = (ob, x, b)
                    assert key not in written, "two ops write one block in a launch"
                    written[key] = True
                    writes.append((ob, x, lo, hi, val))
        assert not (reads & set(written)), "a launch writes a block another op reads"
        for (ob, x, lo, hi, val) in writes:
            if ob == BUF_RANK:
                bufs[BUF_RANK][x][lo:hi] = _round_store(val, dtype).astype(xs[0].dtype)
            else:
                bufs[ob][x][lo:hi] = val
    return bufs[BUF_RANK]


@pytest.mark.parametrize("P,group", [(P, "cyclic") for P in list(range(1, 18)) + [24, 31, 33]]
                         + [(P, "xor") for P in (1, 2, 4, 8, 16, 32)])
def test_step_faithful_tables_reproduce_oracle(P, group):
    rng = np.random.default_rng(P)
    L = G.ceil_log2(P)
    for n in sorted({max(P - 1, 1), 2 * P + 3}):
        for dtype in ("f32", "i32", "bf16"):
            if dtype == "i32":
                xs = [rng.integers(-1000, 1001, n).astype(np.int32) for _ in range(P)]
            else:
                xs = [(rng.standard_normal(n) * np.exp2(rng.integers(-10, 11, n))).astype(np.float32)
                      for _ in range(P)]
                if dtype == "bf16":
                    xs = [G.round_to_bf16(v) for v in xs]
            for S in range(L, 2 * L + 1):
                plan = gar.gar_plan_create_group(P, n, dtype, "sum", S, group)
                got = emulate_step_faithful(plan, xs, dtype, "sum", group)
                want = G.allreduce(xs, S, "sum", dtype, group=group)
                for x in range(P):
                    np.testing.assert_array_equal(got[x].view(np.uint32), want[x].view(np.uint32))


def emulate_fused(plan, xs, op, group="cyclic"):
    P = len(xs)
    n = len(xs[0])
    pairs, outs = gar.gar_plan_fused_program(plan)
    origin = gar.gar_plan_origin(plan)
    t = (lambda b, j: b ^ j) if group == "xor" else (lambda b, j: (b + j) % P)
    res = [np.empty_like(x) for x in xs]
    for b, (lo, hi) in enumerate(_blocks(n, P)):
        vals = [xs[t(b, j)][lo:hi] for j in range(P)]
        for (a, c) in pairs:
            vals.append(_op(op, vals[a], vals[c]))
        for p in range(P):
            res[t(b, p)][lo:hi] = vals[outs[origin[p]]]
    return res


@pytest.mark.parametrize("P,group", [(P, "cyclic") for P in list(range(1, 20)) + [24, 40, 127]]
                         + [(P, "xor") for P in (2, 4, 8, 16, 64, 128)])
def test_fused_program_reproduces_oracle(P, group):
    rng = np.random.default_rng(1000 + P)
    L = G.ceil_log2(P)
    n = 2 * P + 5
    xs = [(rng.standard_normal(n) * np.exp2(rng.integers(-10, 11, n))).astype(np.float32)
          for _ in range(P)]
    for S in range(L, 2 * L + 1):
        for op in ("sum", "max"):
            plan = gar.gar_plan_create_group(P, n, "f32", op, S, group)
            got = emulate_fused(plan, xs, op, group)
            want = G.allreduce(xs, S, op, "f32", group=group)
            for x in range(P):
                np.testing.assert_array_equal(got[x].view(np.uint32), want[x].view(np.uint32))


@pytest.mark.parametrize("P", list(range(4, 18)) + [24, 33])
def test_fold_tables_reproduce_oracle(P):
    """Fold schedules (every even S from 2L+2 to 2(P-1)): the fold counts equal the
    oracle's, and the step-faithful op tables and the fused program reproduce its
    results bit for bit (bf16 sends a never-combined placement in bf16)."""
    rng = np.random.default_rng(700 + P)
    L = G.ceil_log2(P)
    for n in sorted({P - 1, 2 * P + 3}):
        for dtype in ("f32", "i32", "bf16"):
            if dtype == "i32":
                xs = [rng.integers(-1000, 1001, n).astype(np.int32) for _ in range(P)]
            else:
                xs = [(rng.standard_normal(n) * np.exp2(rng.integers(-10, 11, n))).astype(np.float32)
                      for _ in range(P)]
                if dtype == "bf16":
                    xs = [G.round_to_bf16(v) for v in xs]
            for S in range(2 * L + 2, 2 * (P - 1) + 1, 2):
                plan = gar.gar_plan_create(P, n, dtype, "sum", S)
                info = plan.info()
                assert (info["S"], info["K"], info["r"], info["ring"]) == (S, 1, 0, 0)
                assert [len(gar.gar_plan_step(plan, t)[2]) for t in range(S // 2)] == \
                    G.fold_sequence(P, S // 2)
                want = G.allreduce(xs, S, "sum", dtype)
                got = emulate_step_faithful(plan, xs, dtype, "sum")
                for x in range(P):
                    np.testing.assert_array_equal(got[x].view(np.uint32), want[x].view(np.uint32))
                if dtype == "f32":
                    got = emulate_fused(plan, xs, "sum")
                    for x in range(P):
                        np.testing.assert_array_equal(got[x].view(np.uint32), want[x].view(np.uint32))
                if dtype != "bf16":
                    ws, _, _ = gar.gar_plan_bytes(plan)
                    assert ws == 0                # in place, like bandwidth-optimal


def test_fold_argument_errors():
    with pytest.raises(gar.GarError):
        gar.gar_plan_create(24, 10, steps=13)                  # odd S beyond 2L
    with pytest.raises(gar.GarError):
        gar.gar_plan_create(24, 10, steps=48)                  # beyond 2(P-1)
    with pytest.raises(gar.GarError):
        gar.gar_plan_create_group(16, 10, steps=10, group="xor")
    assert gar.gar_plan_create(24, 10, steps=46).info()["S"] == 46


def test_fused_program_size_limit():
    """Fused mode compiles the program as straight-line code and refuses programs over
    GAR_FUSED_MAX_OPS operations (combines + P loads + P stores) at once, with the sizes
    in the message; the step-faithful mode still takes the plan."""
    for (P, S) in [(1024, 10), (1024, 11), (512, 9)]:
        plan = gar.gar_plan_create(P, 5000, "f32", "sum", S)
        ops = plan.info()["fused_combines"] + 2 * P
        assert ops > gar.GAR_FUSED_MAX_OPS
        with pytest.raises(gar.GarError) as e:
            gar.gar_plan_compile(plan, "fused")
        assert e.value.code == -1
        assert f"fused program of {ops} operations" in str(e.value)
        gar.gar_plan_compile(plan, "step")
    # the bandwidth-optimal program at the largest P is within the limit
    plan = gar.gar_plan_create(gar.GAR_MAX_P, 5000, "f32", "sum", gar.GAR_STEPS_BO)
    assert plan.info()["fused_combines"] + 2 * gar.GAR_MAX_P <= gar.GAR_FUSED_MAX_OPS


@pytest.mark.parametrize("P,n,S", [(2, 1, 1), (3, 7, 2), (5, 1031, 3), (24, 5000, 5), (24, 1 << 20, 7),
                                   (24, 1 << 20, 10), (127, 212, 7), (127, 212, 10), (127, 212, 14),
                                   (1000, 5, 10)])
def test_fused_parameter_layout(P, n, S):
    """The generated kernel's gar_args must match the host packing in launch_fused_range:
    in[c P], out[c P], e_lo, e_hi, with c = 2 (tables stored twice) exactly for rotated
    programs with several result copies (1 < K < P) and for single-copy programs over 32
    or more contributions (which also run in 32-thread CTAs), else 1; kernels whose warps
    span several blocks copy the tables to shared memory of the same size."""
    plan = gar.gar_plan_create(P, n, "f32", "sum", S)
    src = gar.gar_plan_fused_source(plan)
    m = re.search(r"struct gar_args \{ const gar_io \*in\[(\d+)\]; gar_io \*out\[(\d+)\]; "
                  r"gar_u64 e_lo, e_hi; \};", src)
    assert m, "unknown parameter layout"
    c = int(m.group(1)) // P
    assert int(m.group(1)) == int(m.group(2)) == c * P and c in (1, 2)
    K = plan.info()["K"]
    small_cta = K == 1 and 32 <= P <= 1000
    assert (c == 2) == (1 < K < P or small_cta)
    assert ("__launch_bounds__(32, 16)" in src) == small_cta
    if "__shared__ const gar_io *s_in[" in src:
        assert K < P                          # only rotated programs stage pointer tables
        assert f"__shared__ const gar_io *s_in[{c * P}];" in src


@pytest.mark.parametrize("P", list(range(2, 41)) + [63, 64, 65, 127, 128])
def test_result_copies_are_shifted_trees(P):
    """Result copy s of the fused program is copy 0's tree with every leaf index shifted
    by s (mod P): the K copies are one schedule shifted by s (cyclic group)."""
    L = G.ceil_log2(P)
    for S in range(L, 2 * L):
        plan = gar.gar_plan_create(P, 1000, "f32", "sum", S)
        pairs, outs = gar.gar_plan_fused_program(plan)
        memo = {}

        def tree(v):
            if v < P:
                return v
            if v not in memo:
                a, b = pairs[v - P]
                memo[v] = (tree(a), tree(b))
            return memo[v]

        def shift(t, s):
            return (t + s) % P if isinstance(t, int) else (shift(t[0], s), shift(t[1], s))

        t0 = tree(outs[0])
        for s in range(len(outs)):
            assert tree(outs[s]) == shift(t0, s), (P, S, s)


def test_workspace_sizes():
    # bandwidth-optimal fp32/int32 runs in place
    for P in (2, 5, 24, 127):
        for dt in ("f32", "i32"):
            ws, _, _ = gar.gar_plan_bytes(gar.gar_plan_create(P, 1000, dt, "sum", gar.GAR_STEPS_BO))
            assert ws == 0
    # bf16 keeps fp32 partials in one slice; other step counts need ping-pong (+ q*)
    ws, _, _ = gar.gar_plan_bytes(gar.gar_plan_create(5, 1000, "bf16", "sum", gar.GAR_STEPS_BO))
    assert ws == 5 * 1024 * 4
    ws, _, _ = gar.gar_plan_bytes(gar.gar_plan_create(8, 1000, "f32", "sum", gar.GAR_STEPS_LO))
    assert ws == 2 * 8 * 1024 * 4          # P = 2^k: q* never separates from q'
    ws, _, _ = gar.gar_plan_bytes(gar.gar_plan_create(7, 1000, "f32", "sum", gar.GAR_STEPS_LO))
    assert ws == 3 * 7 * 1024 * 4


def test_group_argument_errors():
    with pytest.raises(gar.GarError):
        gar.gar_plan_create_group(6, 10, steps=3, group="xor")     # not a power of two
    with pytest.raises(gar.GarError):
        gar.gar_plan_create_group(8, 10, steps=3, group=7)


def test_argument_errors():
    with pytest.raises(gar.GarError) as e:
        gar.gar_plan_create(0, 10)
    assert e.value.code == -1
    with pytest.raises(gar.GarError):
        gar.gar_plan_create(gar.GAR_MAX_P + 1, 10)
    with pytest.raises(gar.GarError):
        gar.gar_plan_create(5, 10, steps=2)          # L = 3
    with pytest.raises(gar.GarError):
        gar.gar_plan_create(5, 10, steps=7)
    with pytest.raises(gar.GarError):
        gar.gar_plan_create(5, 10, dtype=7)
    with pytest.raises(gar.GarError):
        gar.gar_plan_create(5, 10, op=9)
    plan = gar.gar_plan_create(5, 10)
    with pytest.raises(gar.GarError) as e:
        gar.gar_allreduce(plan, [16 * (k + 1) for k in range(4)] + [16 * 3], "fused", stream=0)
    assert e.value.code == -1
    with pytest.raises(gar.GarError) as e:
        gar.gar_allreduce(plan, [16 * (k + 1) + 4 for k in range(5)], "fused", stream=0)
    assert e.value.code == -3
    with pytest.raises(gar.GarError):
        gar.gar_plan_step(plan, 99)
    assert gar.gar_strerror(-3).startswith("buffer")
    # P = 1 and n = 0 are accepted no-ops (no GPU work is launched)
    gar.gar_allreduce(gar.gar_plan_create(1, 10), [64], "fused", stream=0)
    gar.gar_allreduce(gar.gar_plan_create(4, 0), [64, 128, 192, 256], "fused", stream=0)


def test_generated_source_compiles_for_config_shapes():
    for (P, n, dt, S) in [(24, 16777216, "f32", 10), (127, 4194304, "bf16", 7), (127, 4194304, "bf16", 14),
                          (8, 262144, "f32", 4), (5, 1024, "i32", 3)]:
        plan = gar.gar_plan_create(P, n, dt, "sum", S)
        gar.gar_plan_compile(plan, "fused")
        assert plan.info()["fused_width"] >= 1


def test_cost_model_matches_oracle():
    """gar_cost_model / gar_optimal_steps against the oracle's restatement of eqs.
    bo_cost, intemediate_cost, lo_cost and opt_number_of_steps (the oracle's version is
    pinned to the paper's P=127, m=9 KiB example in test_oracle_pins)."""
    import itertools
    params = [(3e-5, 1e-8, 2e-10), (2.5e-6, 1.6e-13, 3e-13), (1e-6, 1e-10, 0.0), (5e-6, 0.0, 1e-12)]
    for P in list(range(1, 40)) + [63, 64, 127, 128, 200]:
        L = G.ceil_log2(P)
        for m in (425.0, 9 * 1024.0, 2 ** 20, 64 * 2 ** 20):
            for (a, b, c) in params:
                for S in range(L, 2 * L + 1):
                    assert gar.gar_cost_model(P, S, m, a, b, c) == pytest.approx(
                        G.cost_model_time(P, m, S, a, b, c), rel=1e-12, abs=1e-300)
                assert gar.gar_optimal_steps(P, m, a, b, c) == G.optimal_steps(P, m, a, b, c)
                # beyond 2L: fold schedules and the Ring; the BO / LO sentinels
                for S in range(2 * L + 2, 2 * (P - 1) + 1, 2):
                    assert gar.gar_cost_model(P, S, m, a, b, c) == pytest.approx(
                        G.cost_model_time(P, m, S, a, b, c), rel=1e-12, abs=1e-300)
                assert gar.gar_cost_model(P, gar.GAR_STEPS_RING, m, a, b, c) == pytest.approx(
                    G.cost_model_time(P, m, "ring", a, b, c), rel=1e-12, abs=1e-300)
                assert gar.gar_cost_model(P, gar.GAR_STEPS_BO, m, a, b, c) == \
                    gar.gar_cost_model(P, 2 * L, m, a, b, c)
                assert gar.gar_cost_model(P, gar.GAR_STEPS_LO, m, a, b, c) == \
                    gar.gar_cost_model(P, L, m, a, b, c)
    with pytest.raises(gar.GarError):
        gar.gar_cost_model(8, 2, 1.0, 1.0, 1.0, 1.0)
    with pytest.raises(gar.GarError):
        gar.gar_cost_model(24, 13, 1.0, 1.0, 1.0, 1.0)     # odd, beyond 2L


@pytest.mark.parametrize("P", [1, 2, 3, 4, 5, 7, 8, 13, 24, 33])
def test_ring_plan_matches_oracle(P):
    """GAR_STEPS_RING: steps, partners, transmitted placements and bytes against the
    oracle's Ring simulation; the op tables and the fused program reproduce its results
    bit for bit on the CPU."""
    rng = np.random.default_rng(500 + P)
    n = 2 * P + 3
    for dtype in ("f32", "bf16", "i32"):
        plan = gar.gar_plan_create(P, n, dtype, "sum", gar.GAR_STEPS_RING)
        run = G.simulate_ring(P, n, dtype=dtype)
        info = plan.info()
        assert info["ring"] == 1 and info["S"] == 2 * (P - 1) == len(run.log)
        _ws, per_step, _S = gar.gar_plan_bytes(plan)
        assert per_step == run.step_bytes()
        for t, st in enumerate(run.log):
            phase, partner, tx = gar.gar_plan_step(plan, t)
            assert phase == (0 if st["phase"] == "reduce" else 1) and partner == -1
            assert tx == [k[0] for k in st["tx"]]
        if dtype == "i32":
            xs = [rng.integers(-1000, 1001, n).astype(np.int32) for _ in range(P)]
        else:
            xs = [(rng.standard_normal(n) * np.exp2(rng.integers(-10, 11, n))).astype(np.float32)
                  for _ in range(P)]
            if dtype == "bf16":
                xs = [G.round_to_bf16(v) for v in xs]
        want = G.simulate_ring(P, n, inputs=xs, dtype=dtype).outputs
        got = emulate_step_faithful(plan, xs, dtype, "sum")
        for x in range(P):
            np.testing.assert_array_equal(got[x].view(np.uint32), want[x].view(np.uint32))
        if dtype == "f32":
            got = emulate_fused(plan, xs, "sum")
            for x in range(P):
                np.testing.assert_array_equal(got[x].view(np.uint32), want[x].view(np.uint32))
    with pytest.raises(gar.GarError):
        gar.gar_plan_create_group(8, 10, "f32", "sum", gar.GAR_STEPS_RING, "xor")


@pytest.mark.parametrize("P,n", [(24, 16777216), (5, 1024), (7, 1001), (127, 4194304), (2, 33)])
def test_bench_dram_model_closed_form(P, n):
    """bench.py's step-faithful DRAM model (bytes the kernels read and write, counted
    from the op tables) against a closed form: bandwidth-optimal fp32 combines every
    element position P - 1 times (partner read + own read + write, 12 B) and copies it
    P - 1 times (read + write, 8 B): (P - 1) * n * 20 bytes.  For P = 24 x 16 Mi that is
    the 7,717,519,360 B the bench reports."""
    import importlib.util
    spec = importlib.util.spec_from_file_location("bench_mod", os.path.join(ROOT, "bench.py"))
    bench = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(bench)
    plan = gar.gar_plan_create(P, n, "f32", "sum", gar.GAR_STEPS_BO)
    assert bench._step_dram_bytes(gar, plan, P, n, "f32") == (P - 1) * n * 20
