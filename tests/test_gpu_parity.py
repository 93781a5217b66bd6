"""GPU parity: libgar's CUDA kernels (through the C ABI) against the CPU oracle.

Floating-point results follow the schedule's association order, so every comparison
with the oracle is bit-exact, for fp32, bf16 (fp32 accumulation) and int32, in both
modes.  Full-size workloads are compared on sampled element positions (the oracle
runs on an element subset) and, everywhere, against properties that hold at any size:
max/min equal the column max/min exactly, and sums lie within the tree error bound
L * 2^-24 * sum|x| of a float64 reference (plus one bf16 rounding, 2^-8 relative).
"""

import numpy as np
import pytest
import torch

import gar_inputs
from oracle import gar_oracle as G

pytestmark = pytest.mark.gpu

gar = pytest.importorskip("paper_2004_09362_gb300.gar")

DEV = "cuda"


def _Ss(P):
    L = G.ceil_log2(P)
    return list(range(L, 2 * L + 1))


def _np_inputs(P, n, dtype, seed, dist=None):
    if dist is None:
        dist = ("int", -1000, 1000) if dtype == "i32" else ("normal", 0.0, 1.0)
    t = gar_inputs.rank_inputs(P, n, dtype, dist, seed)
    return t


def _to_host_list(t, dtype):
    if dtype == "bf16":
        t = t.float()
    return [t[x].numpy().copy() for x in range(t.shape[0])]


def _padded_device(t):
    """Copy a [P, n] tensor to the GPU with a row stride that keeps every row 16-byte
    aligned; returns (storage, row view)."""
    P, n = t.shape
    per16 = 16 // t.element_size()
    n_pad = max(per16, (n + per16 - 1) // per16 * per16)
    store = torch.zeros((P, n_pad), dtype=t.dtype, device=DEV)
    store[:, :n] = t.to(DEV)
    return store, store[:, :n]


def _run(plan, t, mode):
    store, view = _padded_device(t)
    gar.gar_allreduce(plan, store, mode)
    torch.cuda.synchronize()
    return view.cpu()


def _bits(a):
    a = np.ascontiguousarray(a)
    return a.view(np.uint32) if a.dtype.itemsize == 4 else a.view(np.uint16)


def _assert_same(got_t, want_list, dtype, what=""):
    got = _to_host_list(got_t, dtype)
    for x in range(len(want_list)):
        g, w = got[x], want_list[x].astype(got[x].dtype)
        if not np.array_equal(_bits(g), _bits(w)):
            bad = np.nonzero(_bits(g) != _bits(w))[0]
            raise AssertionError(f"{what} rank {x}: {len(bad)} mismatches, first at {bad[:5]}: "
                                 f"got {g[bad[:5]]} want {w[bad[:5]]}")


# ---------------------------------------------------------------------------
# Exhaustive small cases: every P up to 17, every step count, ragged n
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("P", list(range(1, 18)) + [24, 31, 32, 33])
@pytest.mark.parametrize("mode", ["fused", "step"])
def test_small_every_step_count(P, mode):
    """fp32 at ragged sizes around the block and vector boundaries; int32 and bf16 at
    one ragged size; every step count."""
    cases = [(n, "f32") for n in sorted({0, 1, P + 1, 1031})]
    cases += [(4 * P + 3, dt) for dt in ("f32", "i32", "bf16")]
    for (n, dtype) in cases:
        t = _np_inputs(P, n, dtype, seed=P * 1000 + n)
        host = _to_host_list(t, dtype)
        for S in _Ss(P):
            plan = gar.gar_plan_create(P, n, dtype, "sum", S)
            got = _run(plan, t, mode)
            want = G.allreduce(host, S, "sum", dtype)
            _assert_same(got, want, dtype, f"P={P} n={n} {dtype} S={S} {mode}")


@pytest.mark.parametrize("mode", ["fused", "step", "persistent"])
def test_int32_wraparound(mode):
    """int32 sums over the full value range overflow: every mode wraps modulo 2^32 like
    the oracle (two's complement), at ragged small and chunked mid sizes, every S."""
    for (P, n) in [(7, 1001), (24, 24 * 5003 + 11)]:
        rng = np.random.default_rng(P)
        t = torch.from_numpy(rng.integers(-2 ** 31, 2 ** 31, (P, n), dtype=np.int64).astype(np.int32))
        host = _to_host_list(t, "i32")
        for S in _Ss(P):
            plan = gar.gar_plan_create(P, n, "i32", "sum", S)
            _assert_same(_run(plan, t, mode), G.allreduce(host, S, "sum", "i32"), "i32",
                         f"wrap P={P} n={n} S={S} {mode}")


@pytest.mark.parametrize("P", [3, 7, 12])
def test_mid_size_chunked_step_kernel(P):
    """Blocks of ~5000 elements with ragged starts: the chunked step-faithful launch
    (several chunks per block, 16-byte head/tail handling), every step count and type."""
    n = P * 5003 + 5
    for (dtype, op) in (("f32", "sum"), ("i32", "sum"), ("bf16", "sum"), ("bf16", "max")):
        t = _np_inputs(P, n, dtype, seed=33 * P)
        host = _to_host_list(t, dtype)
        for S in _Ss(P):
            plan = gar.gar_plan_create(P, n, dtype, op, S)
            _assert_same(_run(plan, t, "step"), G.allreduce(host, S, op, dtype), dtype,
                         f"P={P} {dtype} {op} S={S}")
            rec = gar.gar_last_step_bytes(plan)
            assert rec == gar.gar_plan_bytes(plan)[1]


@pytest.mark.parametrize("P", range(18, 41))
@pytest.mark.parametrize("mode", ["fused", "step"])
def test_every_p_to_40(P, mode):
    """Every P up to 40 and every step count, fp32, ragged blocks."""
    n = 4 * P + 3
    t = _np_inputs(P, n, "f32", seed=P)
    host = _to_host_list(t, "f32")
    for S in _Ss(P):
        plan = gar.gar_plan_create(P, n, "f32", "sum", S)
        _assert_same(_run(plan, t, mode), G.allreduce(host, S, "sum", "f32"), "f32", f"P={P} S={S} {mode}")


@pytest.mark.parametrize("mode", ["fused", "step", "persistent"])
def test_cuda_graph_capture_and_replay(mode):
    """After gar_plan_prepare, Allreduce calls can be captured into a CUDA graph; each
    replay reduces the buffers' current contents."""
    P, n, S = 7, 7 * 3000 + 5, 4
    t = _np_inputs(P, n, "f32", seed=3)
    plan = gar.gar_plan_create(P, n, "f32", "sum", S)
    if mode != "fused":
        gar.ensure_workspace(plan)
    gar.gar_plan_prepare(plan, "fused" if mode == "fused" else "step")
    store, view = _padded_device(t)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        with torch.cuda.graph(graph, stream=side):
            gar.gar_allreduce(plan, store, mode, side)
    torch.cuda.current_stream().wait_stream(side)
    host = _to_host_list(t, "f32")
    for rep in range(2):
        store[:, :n] = torch.from_numpy(np.stack(host)).to(DEV)
        graph.replay()
        torch.cuda.synchronize()
        _assert_same(view.cpu(), G.allreduce(host, S, "sum", "f32"), "f32", f"graph replay {rep} {mode}")
        host = [h * np.float32(0.5) for h in host]


@pytest.mark.parametrize("op", ["max", "min"])
@pytest.mark.parametrize("mode", ["fused", "step"])
def test_small_max_min(op, mode):
    for P in (2, 3, 5, 6, 7, 8, 12, 13):
        n = 3 * P + 5
        for dtype in ("f32", "i32", "bf16"):
            t = _np_inputs(P, n, dtype, seed=7 * P)
            host = _to_host_list(t, dtype)
            ref = G.column_reduce_exact(host, op, dtype)
            for S in _Ss(P):
                plan = gar.gar_plan_create(P, n, dtype, op, S)
                got = _run(plan, t, mode)
                _assert_same(got, [ref] * P, dtype, f"{op} P={P} {dtype} S={S} {mode}")


# ---------------------------------------------------------------------------
# The paper-shaped workloads at sizes the oracle finishes in seconds
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("mode", ["fused", "step"])
def test_p5_f32_and_i32(mode):
    wl = gar_inputs.WORKLOADS["p5_f32"]
    t = gar_inputs.rank_inputs(wl.P, wl.n, wl.dtype, wl.dist, wl.seed)
    host = _to_host_list(t, "f32")
    for S in wl.steps:
        plan = gar.gar_plan_create(wl.P, wl.n, "f32", "sum", S)
        _assert_same(_run(plan, t, mode), G.allreduce(host, S, "sum", "f32"), "f32", f"S={S}")
    wl = gar_inputs.WORKLOADS["p5_i32"]
    t = gar_inputs.rank_inputs(wl.P, wl.n, wl.dtype, wl.dist, wl.seed)
    host = _to_host_list(t, "i32")
    for op in wl.ops:
        for S in wl.steps:
            plan = gar.gar_plan_create(wl.P, wl.n, "i32", op, S)
            _assert_same(_run(plan, t, mode), G.allreduce(host, S, op, "i32"), "i32", f"{op} S={S}")


@pytest.mark.parametrize("mode", ["fused", "step"])
def test_p8_1mib_every_step_count(mode):
    wl = gar_inputs.WORKLOADS["p8_1mib_f32"]
    t = gar_inputs.rank_inputs(wl.P, wl.n, wl.dtype, wl.dist, wl.seed)
    host = _to_host_list(t, "f32")
    for S in wl.steps:
        plan = gar.gar_plan_create(wl.P, wl.n, "f32", "sum", S)
        _assert_same(_run(plan, t, mode), G.allreduce(host, S, "sum", "f32"), "f32", f"S={S}")


@pytest.mark.parametrize("mode", ["fused", "step"])
def test_p127_bf16_reduced_n(mode):
    """P=127 bf16 with fp32 accumulation at a ragged n that spans several vector widths
    per block; every step count 7..14."""
    P, n = 127, 127 * 40 + 19
    t = gar_inputs.rank_inputs(P, n, "bf16", ("normal", 0.0, 1.0), 99)
    host = _to_host_list(t, "bf16")
    for S in range(7, 15):
        plan = gar.gar_plan_create(P, n, "bf16", "sum", S)
        _assert_same(_run(plan, t, mode), G.allreduce(host, S, "sum", "bf16"), "bf16", f"S={S}")


@pytest.mark.parametrize("P,n,dtype", [(32, 32 * 40000 + 13, "bf16"), (64, 1 << 20, "f32"),
                                       (48, 48 * 2048 * 3 + 100, "i32")])
def test_latency_optimal_mid_size_fused(P, n, dtype):
    """Latency-optimal programs with P = 32..64 (hundreds of combines per element
    position, every rank its own tree rotation) at sizes with ragged tails, checked on
    sampled positions."""
    t = _np_inputs(P, n, dtype, seed=P)
    plan = gar.gar_plan_create(P, n, dtype, "sum", gar.GAR_STEPS_LO)
    got = _run(plan, t, "fused")
    idx = _sample(n, P, k=2048, seed=P)
    full = [np.zeros(n, np.float32 if dtype != "i32" else np.int32) for _ in range(P)]
    host = _to_host_list(t, dtype)
    for x in range(P):
        full[x][idx] = host[x][idx]
    want = G.allreduce(full, G.ceil_log2(P), "sum", dtype, elements=idx)
    gotl = _to_host_list(got, dtype)
    for x in range(P):
        g = gotl[x][idx].astype(want[x].dtype)
        assert np.array_equal(_bits(g), _bits(want[x])), f"rank {x}"


# ---------------------------------------------------------------------------
# The breadth-first fused form (step by step, paired fp32 adds, bf16 mixed adds)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("P,n", [(40, 40 * 97 + 13), (127, 127 * 40 + 19), (127, 3 * 127 + 5)])
@pytest.mark.parametrize("dtype,op", [("f32", "sum"), ("bf16", "sum"), ("i32", "sum"), ("f32", "max")])
def test_breadth_first_form_every_step_count(P, n, dtype, op, monkeypatch):
    """The breadth-first form forced on for every step count with several result copies
    (it is the default only for large float sums at small S), bit for bit against the
    oracle; n = 3P + 5 puts several blocks in one warp (pointer tables in shared memory)."""
    monkeypatch.setenv("GAR_TUNE_FUSED_FORM", "1")
    t = _np_inputs(P, n, dtype, seed=P + n)
    host = _to_host_list(t, dtype)
    L = G.ceil_log2(P)
    for S in range(L, 2 * L):
        plan = gar.gar_plan_create(P, n, dtype, op, S)
        assert gar.gar_plan_get_info(plan)["fused_form"] == gar.GAR_FORM_BREADTH
        _assert_same(_run(plan, t, "fused"), G.allreduce(host, S, op, dtype), dtype, f"S={S}")


@pytest.mark.parametrize("P,n", [(40, 40 * 97 + 13), (127, 127 * 40 + 19), (127, 3 * 127 + 5), (64, 64 * 33 + 1),
                                 (5, 1000), (24, 24 * 16 + 15)])
@pytest.mark.parametrize("dtype,op", [("f32", "sum"), ("bf16", "sum"), ("i32", "sum"), ("f32", "max"), ("bf16", "min")])
def test_two_lane_form_latency_optimal(P, n, dtype, op, monkeypatch):
    """The two-lane form forced on for the latency-optimal schedule, bit for bit against
    the oracle; odd and even P, ragged n (the last warp's group of 16 positions is
    partial)."""
    monkeypatch.setenv("GAR_TUNE_FUSED_FORM", "2")
    t = _np_inputs(P, n, dtype, seed=3 * P + n)
    host = _to_host_list(t, dtype)
    S = G.ceil_log2(P)
    plan = gar.gar_plan_create(P, n, dtype, op, S)
    assert gar.gar_plan_get_info(plan)["fused_form"] == gar.GAR_FORM_SPLIT
    _assert_same(_run(plan, t, "fused"), G.allreduce(host, S, op, dtype), dtype, f"P={P} S={S}")


def test_register_heavy_single_kernels_get_small_ctas():
    """Once prepared, a single-thread kernel of more than 128 registers runs in 64-thread
    CTAs capped at 168 registers; where that build spills more than 256 bytes per thread,
    32-thread CTAs with up to 255 registers replace it if they spill less; lighter kernels
    keep 256-thread CTAs."""
    heavy = gar.gar_plan_create(127, 4194304, "bf16", "sum", 9)
    gar.gar_plan_prepare(heavy, "fused")
    info = gar.gar_plan_get_info(heavy)
    src = gar.gar_plan_fused_source(heavy)
    if "__launch_bounds__(64, 5)" in src:
        assert info["fused_regs"] <= 168 and info["fused_local_bytes"] <= 256
    else:
        assert "__launch_bounds__(32, 8)" in src
    spilling = gar.gar_plan_create(127, 4194304, "bf16", "sum", 10)
    gar.gar_plan_prepare(spilling, "fused")
    src = gar.gar_plan_fused_source(spilling)
    assert "__launch_bounds__(64, 5)" in src or "__launch_bounds__(32, 8)" in src
    if "__launch_bounds__(32, 8)" in src:
        assert gar.gar_plan_get_info(spilling)["fused_regs"] > 168
    light = gar.gar_plan_create(24, 1 << 24, "f32", "sum", 10)
    gar.gar_plan_prepare(light, "fused")
    assert "__launch_bounds__(256)" in gar.gar_plan_fused_source(light)


@pytest.mark.parametrize("P", [8, 32])
def test_breadth_first_form_xor_group(P, monkeypatch):
    monkeypatch.setenv("GAR_TUNE_FUSED_FORM", "1")
    n = 5 * P + 3
    t = _np_inputs(P, n, "f32", seed=P)
    host = _to_host_list(t, "f32")
    L = G.ceil_log2(P)
    for S in range(L, 2 * L):
        plan = gar.gar_plan_create_group(P, n, "f32", "sum", S, "xor")
        _assert_same(_run(plan, t, "fused"), G.allreduce(host, S, "sum", "f32", group="xor"), "f32", f"S={S}")


# ---------------------------------------------------------------------------
# Recorded step bytes equal the schedule's predicted volume
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("P,n,dtype", [(5, 1024, "f32"), (8, 262144, "f32"), (7, 1001, "bf16"),
                                       (24, 24 * 1000 + 7, "f32"), (127, 5000, "bf16")])
def test_recorded_step_bytes(P, n, dtype):
    t = _np_inputs(P, n, dtype, seed=5)
    for S in _Ss(P):
        plan = gar.gar_plan_create(P, n, dtype, "sum", S)
        _run(plan, t, "step")
        rec = gar.gar_last_step_bytes(plan)
        _ws, pred, _S = gar.gar_plan_bytes(plan)
        run = G.simulate(P, n, S, dtype=dtype)
        assert rec == pred == run.step_bytes(), (P, S, rec, pred)


# ---------------------------------------------------------------------------
# Full sizes, in the launch configuration bench.py times
# ---------------------------------------------------------------------------

def _sample(n, P, k=4096, seed=0):
    rng = np.random.default_rng(seed)
    bounds = G.block_bounds(n, P)
    picks = [rng.integers(0, n, k)]
    for (lo, hi) in bounds:                       # both ends of every block
        if hi > lo:
            picks.append(np.array([lo, min(lo + 1, hi - 1), max(hi - 2, lo), hi - 1]))
    picks.append(np.array([0, n - 1]))
    return np.unique(np.concatenate(picks))


def _tree_bound_check(got_rows, inp, L, dtype):
    """Property at any size: |result - exact| <= L 2^-24 sum|x| (+ 2^-8 |exact| for bf16)."""
    x64 = inp.to(DEV, torch.float64)
    exact = x64.sum(0)
    mag = x64.abs().sum(0)
    tol = L * 2.0 ** -24 * mag * 1.0001
    if dtype == "bf16":
        tol = tol + 2.0 ** -8 * exact.abs()
    for r in range(got_rows.shape[0]):
        err = (got_rows[r].to(torch.float64) - exact).abs()
        assert bool((err <= tol + 1e-30).all()), f"rank {r}: max excess {(err - tol).max().item()}"


def _kahan_check(got_rows, inp, rtol):
    """The stated float tolerance: |result - ref| <= rtol * sum_j |x_j| per element, ref
    the compensated (Kahan) sum of the P inputs in rank order, in float64 on the device;
    rtol 1e-6 for fp32, 1e-2 for bf16 (fp32 accumulation, one final rounding)."""
    s = torch.zeros(inp.shape[1], dtype=torch.float64, device=DEV)
    c = torch.zeros_like(s)
    mag = torch.zeros_like(s)
    for j in range(inp.shape[0]):
        xj = inp[j].to(DEV, torch.float64)
        y = xj - c
        t = s + y
        c = (t - s) - y
        s = t
        mag += xj.abs()
    tol = rtol * mag
    for r in range(got_rows.shape[0]):
        err = (got_rows[r].to(torch.float64) - s).abs()
        assert bool((err <= tol).all()), f"rank {r}: max excess {(err - tol).max().item()}"


@pytest.mark.parametrize("S", [10, 22, 46])
@pytest.mark.parametrize("mode", ["fused", "step"])
def test_full_p24_64mib(S, mode):
    """The 24 x 64 MiB fp32 workload: bandwidth-optimal (S = 10) and two fold schedules
    (S = 22, and S = 46 = 2(P-1), one vector folded per step)."""
    wl = gar_inputs.WORKLOADS["p24_64mib_f32"]
    P, n = wl.P, wl.n
    inp = gar_inputs.rank_inputs(P, n, wl.dtype, wl.dist, wl.seed, device=DEV)
    buf = inp.clone()
    plan = gar.gar_plan_create(P, n, "f32", "sum", S)
    gar.gar_allreduce(plan, buf, mode)
    torch.cuda.synchronize()
    # one result copy: every rank holds identical bits
    assert bool((buf == buf[0:1]).all())
    # the result tree's depth is the number of reduction steps
    _tree_bound_check(buf, inp, S // 2, "f32")
    _kahan_check(buf, inp, 1e-6)
    idx = _sample(n, P)
    host_in = [inp[x, torch.from_numpy(idx).to(DEV)].cpu().numpy() for x in range(P)]
    # oracle on the sampled element positions: rebuild full-length vectors lazily by
    # running it on the subset (elementwise => exact)
    full = [np.zeros(n, np.float32) for _ in range(P)]
    for x in range(P):
        full[x][idx] = host_in[x]
    want = G.allreduce(full, S, "sum", "f32", elements=idx)
    got = buf[:, torch.from_numpy(idx).to(DEV)].cpu().numpy()
    for x in range(P):
        np.testing.assert_array_equal(got[x].view(np.uint32), want[x].view(np.uint32))
    if mode == "step":
        rec = gar.gar_last_step_bytes(plan)
        _ws, pred, _S = gar.gar_plan_bytes(plan)
        assert rec == pred


@pytest.mark.parametrize("S", list(range(7, 15)))
@pytest.mark.parametrize("mode", ["fused", "step"])
def test_full_p127_8mib_bf16(S, mode):
    wl = gar_inputs.WORKLOADS["p127_8mib_bf16"]
    P, n = wl.P, wl.n
    inp = gar_inputs.rank_inputs(P, n, wl.dtype, wl.dist, wl.seed, device=DEV)
    buf = inp.clone()
    plan = gar.gar_plan_create(P, n, "bf16", "sum", S)
    gar.gar_allreduce(plan, buf, mode)
    torch.cuda.synchronize()
    _tree_bound_check(buf.float(), inp.float(), 7, "bf16")
    _kahan_check(buf.float(), inp.float(), 1e-2)
    idx = _sample(n, P, k=512, seed=S)
    sel = torch.from_numpy(idx).to(DEV)
    sub = inp[:, sel].float().cpu().numpy()
    full = [np.zeros(n, np.float32) for _ in range(P)]
    for x in range(P):
        full[x][idx] = sub[x]
    want = G.allreduce(full, S, "sum", "bf16", elements=idx)
    got = buf[:, sel].float().cpu().numpy()
    for x in range(P):
        np.testing.assert_array_equal(got[x].view(np.uint32), want[x].view(np.uint32))


# ---------------------------------------------------------------------------
# Batched small Allreduces (65536 instances of P=6 / P=7, 106 fp32 per rank)
# ---------------------------------------------------------------------------

def _batched_setup(count, Ps, n, seed, op, steps="lo"):
    flat, layout = gar_inputs.batched_inputs(count, Ps, n, "f32", ("normal", 0.0, 1.0), seed,
                                             device=DEV)
    out = torch.empty_like(flat)
    plans = [gar.gar_plan_create(P, n, "f32", op, gar.GAR_STEPS_LO if steps == "lo" else steps)
             for P in Ps]
    idx = {P: k for k, P in enumerate(Ps)}
    es = flat.element_size()
    desc = gar.make_batch_desc([idx[P] for (P, _o) in layout],
                               [flat.data_ptr() + o * es for (_P, o) in layout],
                               [out.data_ptr() + o * es for (_P, o) in layout])
    return flat, out, layout, plans, desc


@pytest.mark.parametrize("op", ["sum", "max"])
def test_batched_425_bytes(op):
    count, Ps, n = 65536, (6, 7), 106
    flat, out, layout, plans, desc = _batched_setup(count, Ps, n, 1236, op)
    gar.gar_allreduce_batched(plans, desc, count)
    torch.cuda.synchronize()
    rng = np.random.default_rng(1)
    check = np.unique(np.concatenate([[0, count // 2 - 1, count // 2, count - 1],
                                      rng.integers(0, count, 200)]))
    fh, oh = flat.cpu().numpy(), out.cpu().numpy()
    for i in check:
        P, off = layout[i]
        xs = [fh[off + x * n: off + (x + 1) * n].copy() for x in range(P)]
        want = G.allreduce(xs, G.ceil_log2(P), op, "f32")
        for x in range(P):
            got = oh[off + x * n: off + (x + 1) * n]
            np.testing.assert_array_equal(got.view(np.uint32), want[x].view(np.uint32))
    # every instance: property check against float64 / exact max
    for P in Ps:
        offs = np.array([o for (p, o) in layout if p == P])
        base = torch.from_numpy(offs).to(DEV)
        ar = torch.arange(P * n, device=DEV)
        gi = (base[:, None] + ar[None, :]).view(-1, P, n)
        xin, xout = flat[gi], out[gi]
        if op == "max":
            assert bool((xout == xin.max(1, keepdim=True).values).all())
        else:
            x64 = xin.double()
            tol = 3 * 2.0 ** -24 * x64.abs().sum(1, keepdim=True) * 1.0001
            assert bool(((xout.double() - x64.sum(1, keepdim=True)).abs() <= tol + 1e-30).all())


def test_batched_mixed_order_and_steps():
    """Instances of different plans interleaved, intermediate step counts, in == out, and
    a misaligned instance (handled element-wise)."""
    n = 50
    Ps = (3, 5, 6)
    plans = [gar.gar_plan_create(3, n, "f32", "sum", 3), gar.gar_plan_create(5, n, "f32", "sum", 4),
             gar.gar_plan_create(6, n, "f32", "sum", 5)]
    count = 300
    rng = np.random.default_rng(3)
    which = rng.integers(0, 3, count)
    sizes = [Ps[w] * n for w in which]
    offs = np.concatenate([[0], np.cumsum(sizes)])[:-1] + 1    # +1 element: misaligned base
    data = torch.randn(int(offs[-1] + sizes[-1] + 8), device=DEV)
    ref_in = data.cpu().numpy().copy()
    es = 4
    desc = gar.make_batch_desc(which, [data.data_ptr() + int(o) * es for o in offs],
                               [data.data_ptr() + int(o) * es for o in offs])
    gar.gar_allreduce_batched(plans, desc, count)
    torch.cuda.synchronize()
    got = data.cpu().numpy()
    steps = (3, 4, 5)
    for i in range(count):
        P, o, S = Ps[which[i]], int(offs[i]), steps[which[i]]
        xs = [ref_in[o + x * n: o + (x + 1) * n].copy() for x in range(P)]
        want = G.allreduce(xs, S, "sum", "f32")
        for x in range(P):
            np.testing.assert_array_equal(got[o + x * n: o + (x + 1) * n].view(np.uint32),
                                          want[x].view(np.uint32))


# ---------------------------------------------------------------------------
# The XOR group (Table 1b): Recursive Halving / Doubling and their hybrids
# ---------------------------------------------------------------------------

def _run_group(P, n, dtype, S, mode, t, group):
    plan = gar.gar_plan_create_group(P, n, dtype, "sum", S, group)
    return plan, _run(plan, t, mode)


@pytest.mark.parametrize("P", [2, 4, 8, 16, 32, 64])
@pytest.mark.parametrize("mode", ["fused", "step", "persistent"])
def test_xor_group_matches_oracle(P, mode):
    cases = [(2 * P + 3, "f32"), (2 * P + 3, "i32"), (2 * P + 3, "bf16"), (P * 4099 + 1, "f32")]
    for (n, dtype) in cases:
        t = _np_inputs(P, n, dtype, seed=17 * P + n)
        host = _to_host_list(t, dtype)
        for S in _Ss(P):
            plan, got = _run_group(P, n, dtype, S, mode, t, "xor")
            _assert_same(got, G.allreduce(host, S, "sum", dtype, group="xor"), dtype,
                         f"xor P={P} n={n} {dtype} S={S} {mode}")
            if mode != "fused":
                assert gar.gar_last_step_bytes(plan) == gar.gar_plan_bytes(plan)[1]


def test_batched_mixed_groups():
    n = 64
    plans = [gar.gar_plan_create_group(8, n, "f32", "sum", 4, "xor"),
             gar.gar_plan_create_group(6, n, "f32", "sum", 4, "cyclic"),
             gar.gar_plan_create_group(16, n, "f32", "sum", 4, "xor")]
    Ps, steps, groups = (8, 6, 16), (4, 4, 4), ("xor", "cyclic", "xor")
    count = 90
    which = [i % 3 for i in range(count)]
    sizes = [Ps[w] * n for w in which]
    offs = np.concatenate([[0], np.cumsum(sizes)])[:-1]
    data = torch.randn(int(offs[-1] + sizes[-1]), device=DEV)
    ref_in = data.cpu().numpy().copy()
    desc = gar.make_batch_desc(which, [data.data_ptr() + int(o) * 4 for o in offs],
                               [data.data_ptr() + int(o) * 4 for o in offs])
    gar.gar_allreduce_batched(plans, desc, count)
    torch.cuda.synchronize()
    got = data.cpu().numpy()
    for i in range(count):
        w, o = which[i], int(offs[i])
        P = Ps[w]
        xs = [ref_in[o + x * n: o + (x + 1) * n].copy() for x in range(P)]
        want = G.allreduce(xs, steps[w], "sum", "f32", group=groups[w])
        for x in range(P):
            np.testing.assert_array_equal(got[o + x * n: o + (x + 1) * n].view(np.uint32),
                                          want[x].view(np.uint32))


@pytest.mark.parametrize("P", [2, 3, 5, 8, 24])
@pytest.mark.parametrize("mode", ["fused", "step", "persistent"])
def test_ring_matches_oracle(P, mode):
    """The Ring schedule (2(P-1) steps) bit for bit against the oracle's Ring."""
    for (n, dtype) in [(2 * P + 3, "f32"), (2 * P + 3, "bf16"), (2 * P + 3, "i32"), (P * 4001 + 3, "f32")]:
        t = _np_inputs(P, n, dtype, seed=29 * P + n)
        host = _to_host_list(t, dtype)
        plan = gar.gar_plan_create(P, n, dtype, "sum", gar.GAR_STEPS_RING)
        got = _run(plan, t, mode)
        _assert_same(got, G.allreduce(host, "ring", "sum", dtype), dtype, f"ring P={P} n={n} {dtype} {mode}")
        if mode != "fused":
            assert gar.gar_last_step_bytes(plan) == gar.gar_plan_bytes(plan)[1]


def _fold_Ss(P):
    L = G.ceil_log2(P)
    return list(range(2 * L + 2, 2 * (P - 1) + 1, 2))


@pytest.mark.parametrize("P", [4, 5, 7, 8, 13, 24])
@pytest.mark.parametrize("mode", ["fused", "step", "persistent"])
def test_fold_schedules_match_oracle(P, mode):
    """Fold schedules (every even S from 2L+2 to 2(P-1)) bit for bit against the oracle:
    ragged small blocks in three types and with max, mid-size blocks (chunked step
    launch) in fp32 and bf16; recorded step bytes equal the prediction."""
    cases = [(2 * P + 3, "f32", "sum"), (2 * P + 3, "bf16", "sum"), (2 * P + 3, "i32", "sum"),
             (2 * P + 3, "f32", "max"), (P * 4001 + 3, "f32", "sum"), (P * 2001 + 5, "bf16", "sum")]
    for (n, dtype, op) in cases:
        t = _np_inputs(P, n, dtype, seed=41 * P + n)
        host = _to_host_list(t, dtype)
        for S in _fold_Ss(P):
            plan = gar.gar_plan_create(P, n, dtype, op, S)
            got = _run(plan, t, mode)
            _assert_same(got, G.allreduce(host, S, op, dtype), dtype,
                         f"fold P={P} n={n} {dtype} {op} S={S} {mode}")
            if mode != "fused":
                assert gar.gar_last_step_bytes(plan) == gar.gar_plan_bytes(plan)[1]
            if mode == "persistent":
                assert gar.gar_plan_status(plan) == 0


# ---------------------------------------------------------------------------
# Persistent step-faithful mode: one cooperative launch, bounded grid barriers
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("P", [2, 5, 7, 8, 13, 24, 33])
def test_persistent_matches_oracle(P):
    """Small blocks (element-major mapping) and mid-size blocks (chunked mapping),
    every step count, all three types; recorded step bytes; no barrier timeout."""
    for n in (3 * P + 1, P * 3001 + 7):
        for dtype in ("f32", "i32", "bf16"):
            if n > 1000 and dtype != "f32" and P not in (7, 24):
                continue
            t = _np_inputs(P, n, dtype, seed=5 * P + n)
            host = _to_host_list(t, dtype)
            for S in _Ss(P):
                plan = gar.gar_plan_create(P, n, dtype, "sum", S)
                got = _run(plan, t, "persistent")
                assert gar.gar_plan_status(plan) == 0
                _assert_same(got, G.allreduce(host, S, "sum", dtype), dtype,
                             f"persistent P={P} n={n} {dtype} S={S}")
                assert gar.gar_last_step_bytes(plan) == gar.gar_plan_bytes(plan)[1]


def test_persistent_barrier_timeout_is_reported_and_recoverable():
    """Make every grid-barrier wait run out (the barrier waits for one CTA that was never
    launched): the kernel returns on its own, gar_plan_status reports GAR_ETIMEOUT, and
    the same context then runs correct Allreduces."""
    P, n, S = 7, 5000, 4
    t = _np_inputs(P, n, "f32", seed=1)
    plan = gar.gar_plan_create(P, n, "f32", "sum", S)
    gar.gar_plan_debug_barrier(plan, phantom=1, spin_limit=2000)
    _run(plan, t, "persistent")
    assert gar.gar_plan_status(plan) == -8
    assert "gave up" in gar.gar_last_error()
    gar.gar_plan_debug_barrier(plan, phantom=0, spin_limit=0)
    want = G.allreduce(_to_host_list(t, "f32"), S, "sum", "f32")
    _assert_same(_run(plan, t, "persistent"), want, "f32", "after timeout")
    assert gar.gar_plan_status(plan) == 0
    _assert_same(_run(plan, t, "fused"), want, "f32", "fused after timeout")


# ---------------------------------------------------------------------------
# Host-buffer entry point and argument handling on the device
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("layout", ["pinned", "pinned_misaligned", "pageable"])
@pytest.mark.parametrize("P,n,dtype,S", [(7, 70001, "f32", 4), (5, 16 * 65536 + 37, "bf16", 5),
                                         (24, 3 * 65536 + 5, "f32", 10), (6, 1000, "i32", 3)])
@pytest.mark.parametrize("mode", ["fused", "step"])
def test_host_buffers(P, n, dtype, S, mode, layout):
    """gar_allreduce_host.  Fused mode on aligned host memory the GPU can address runs
    the kernel on the host buffers directly; misaligned host rows take the staged path
    (copies in element chunks pipelined over internal streams, several chunks and a
    ragged last chunk here); step-faithful mode copies, reduces, copies back."""
    t = _np_inputs(P, n, dtype, seed=11)
    off = 1 if layout == "pinned_misaligned" else 0
    host_in = torch.zeros((P, n + off), dtype=t.dtype)
    host_in[:, off:] = t
    host_out = torch.zeros_like(host_in)
    if layout != "pageable":
        host_in, host_out = host_in.pin_memory(), host_out.pin_memory()
    dev_store, _ = _padded_device(t)
    plan = gar.gar_plan_create(P, n, dtype, "sum", S)
    rows_in = [host_in[x, off:] for x in range(P)]
    rows_out = [host_out[x, off:] for x in range(P)]
    gar.gar_allreduce_host(plan, rows_in, rows_out, dev_store, mode)
    torch.cuda.synchronize()
    want = G.allreduce(_to_host_list(t, dtype), S, "sum", dtype)
    _assert_same(host_out[:, off:], want, dtype, "host")
    assert bool((host_in[:, off:] == t).all())        # inputs untouched


@pytest.mark.parametrize("mode", ["fused", "step", "persistent"])
def test_host_buffers_other_schedules(mode):
    """gar_allreduce_host with every schedule family: a fold schedule, the Ring and the
    XOR group (pinned, aligned rows), and persistent mode on the copy path."""
    for (P, n, dtype, steps, group, want_S) in [(24, 24 * 3001 + 5, "f32", 22, "cyclic", 22),
                                                (8, 8 * 2001 + 3, "bf16", gar.GAR_STEPS_RING, "cyclic", "ring"),
                                                (16, 16 * 4001, "f32", 6, "xor", 6)]:
        t = _np_inputs(P, n, dtype, seed=17 + P)
        per16 = 16 // t.element_size()
        n_pad = (n + per16 - 1) // per16 * per16
        host_in = torch.zeros((P, n_pad), dtype=t.dtype)
        host_in[:, :n] = t
        host_out = torch.zeros_like(host_in)
        host_in, host_out = host_in.pin_memory(), host_out.pin_memory()
        dev_store, _ = _padded_device(t)
        plan = gar.gar_plan_create_group(P, n, dtype, "sum", steps, group)
        rows_in = [host_in[x, :n] for x in range(P)]
        rows_out = [host_out[x, :n] for x in range(P)]
        gar.gar_allreduce_host(plan, rows_in, rows_out, dev_store, mode)
        torch.cuda.synchronize()
        want = G.allreduce(_to_host_list(t, dtype), want_S, "sum", dtype, group=group)
        _assert_same(host_out[:, :n], want, dtype, f"host P={P} {group} S={want_S} {mode}")
        assert bool((host_in[:, :n] == t).all())


def test_missing_workspace_is_an_error():
    P, n = 7, 100
    plan = gar.gar_plan_create(P, n, "f32", "sum", 3)
    store, _ = _padded_device(torch.zeros(P, n))
    import ctypes
    ptrs = (ctypes.c_void_p * P)(*[store[x].data_ptr() for x in range(P)])
    rc = gar._lib.gar_allreduce(plan.handle, ptrs, gar.GAR_STEP_FAITHFUL,
                                ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == -6
