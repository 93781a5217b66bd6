"""Property-based check of the schedule builder against the oracle (CPU, no GPU):
random P (up to 200), random step count in the plan's whole range (including fold
schedules and the Ring), both groups, all element types and operators, ragged n.  The
step-faithful op tables and the fused program, executed on the CPU with the kernels'
semantics, must give the oracle's bits at every rank."""

import numpy as np
import pytest

from oracle import gar_oracle as G
from paper_2004_09362_gb300 import gar

hyp = pytest.importorskip("hypothesis")
st = hyp.strategies

from test_plan_host import emulate_fused, emulate_step_faithful  # noqa: E402


@st.composite
def plans(draw):
    P = draw(st.integers(1, 200))
    L = G.ceil_log2(P)
    xor = P & (P - 1) == 0 and P > 1 and draw(st.booleans())
    choices = list(range(L, 2 * L + 1))
    if not xor and P > 2:
        choices += list(range(2 * L + 2, 2 * (P - 1) + 1, 2)) + ["ring"]
    S = draw(st.sampled_from(choices))
    n = draw(st.integers(0, 3 * P + 7))
    dtype = draw(st.sampled_from(["f32", "i32", "bf16"]))
    op = draw(st.sampled_from(["sum", "max", "min"]))
    seed = draw(st.integers(0, 2 ** 31 - 1))
    return P, S, n, dtype, op, ("xor" if xor else "cyclic"), seed


@hyp.settings(max_examples=80, deadline=None, derandomize=True)
@hyp.given(plans())
def test_random_plans_reproduce_oracle(case):
    P, S, n, dtype, op, group, seed = case
    rng = np.random.default_rng(seed)
    if dtype == "i32":
        xs = [rng.integers(-2 ** 31, 2 ** 31, n, dtype=np.int64).astype(np.int32) for _ in range(P)]
    else:
        xs = [(rng.standard_normal(n) * np.exp2(rng.integers(-12, 13, n))).astype(np.float32)
              for _ in range(P)]
        if dtype == "bf16":
            xs = [G.round_to_bf16(v) for v in xs]
    steps = gar.GAR_STEPS_RING if S == "ring" else S
    plan = gar.gar_plan_create_group(P, n, dtype, op, steps, group)
    want = G.allreduce(xs, S, op, dtype, group=group)
    got = emulate_step_faithful(plan, xs, dtype, op, group)
    for x in range(P):
        np.testing.assert_array_equal(got[x].view(np.uint32), want[x].view(np.uint32))
    if dtype == "f32":
        got = emulate_fused(plan, xs, op, group)
        for x in range(P):
            np.testing.assert_array_equal(got[x].view(np.uint32), want[x].view(np.uint32))
