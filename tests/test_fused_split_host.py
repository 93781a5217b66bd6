"""Host-side checks of the two-lane fused kernel (GAR_FORM_SPLIT, no GPU).

In this form two lanes of a warp share an element position: lane half A evaluates the
combines at placements [0, m), half B the same code rotated by m placements, and the
vectors a step moves across the halves arrive by a warp shuffle.  These tests check,
without a GPU:
  * which plans the form applies to (rotation-invariant, latency-optimal cyclic);
  * that its generated evaluation code, run for both halves in lockstep by a small
    interpreter written here in numpy float32 (the shuffle swaps the halves' values),
    gives the oracle's bits for every rank and element;
  * that a planted mistake in the exchange is caught;
  * that NVRTC compiles it for sm_103a.
"""

import os
import re

import numpy as np
import pytest

from oracle import gar_oracle as O
from paper_2004_09362_gb300 import gar as G


def _split_source(P, n, dtype, S, op="sum"):
    old = os.environ.get("GAR_TUNE_FUSED_FORM")
    os.environ["GAR_TUNE_FUSED_FORM"] = "2"
    try:
        pl = G.gar_plan_create(P, n, dtype, op, S)
        return G.gar_plan_fused_source(pl), G.gar_plan_get_info(pl)
    finally:
        if old is None:
            os.environ.pop("GAR_TUNE_FUSED_FORM", None)
        else:
            os.environ["GAR_TUNE_FUSED_FORM"] = old


def _bf16_round(x):
    return O.round_to_bf16(np.asarray(x, dtype=np.float32))


def _run_split(src, P, xs, dtype, op):
    """Evaluates gar_eval_sp for every element of P rank vectors xs, both lane halves
    statement by statement; returns the P output vectors."""
    body = re.search(r"void gar_eval_sp\(.*?\{\n(.*?)\n\}\n", src, re.S).group(1)
    m = int(re.search(r"s_in \+ \(hb \? (\d+) : 0\)", src).group(1))
    n = len(xs[0])
    comb = {"sum": lambda a, c: np.float32(a + c), "max": lambda a, c: np.float32(max(a, c)),
            "min": lambda a, c: np.float32(min(a, c))}[op]
    if dtype == "i32":
        comb = {"sum": lambda a, c: np.int32((int(a) + int(c) + 2**31) % 2**32 - 2**31),
                "max": lambda a, c: max(a, c), "min": lambda a, c: min(a, c)}[op]
    out = [np.zeros_like(x) for x in xs]
    written = [np.zeros(n, dtype=int) for _ in range(P)]
    lines = [ln.strip() for ln in body.split("\n") if ln.strip() and not ln.strip().startswith("(void)")]
    for e in range(n):
        env = [{}, {}]

        def val(h, tok):
            tok = tok.strip()
            mm = re.fullmatch(r"gar_wide\(([ly]\d+)\)", tok)
            return env[h][mm.group(1)] if mm else env[h][tok]

        for ln in lines:
            mm = re.fullmatch(r"const gar_io (l\d+) = gar_ldio\(tin\[(\d+)\] \+ e\);", ln)
            if mm:
                for h in (0, 1):
                    env[h][mm.group(1)] = xs[(h * m + int(mm.group(2))) % P][e]
                continue
            mm = re.fullmatch(r"const gar_(?:io|acc) ([xy]\d+) = gar_x(?:io|acc)\(hb \? (\w+) : (\w+)\);", ln)
            if mm:
                send = [env[0][mm.group(3)], env[1][mm.group(2)]]   # hb = 0 sends the second
                env[0][mm.group(1)], env[1][mm.group(1)] = send[1], send[0]
                continue
            mm = re.fullmatch(r"const float2 (w\d+) = __fadd2_rn\(make_float2\((.*), (.*)\), make_float2\((.*), (.*)\)\);", ln)
            if mm:
                for h in (0, 1):
                    env[h][mm.group(1)] = (np.float32(val(h, mm.group(2)) + val(h, mm.group(4))),
                                           np.float32(val(h, mm.group(3)) + val(h, mm.group(5))))
                continue
            mm = re.fullmatch(r"const gar_acc (v\d+) = (w\d+)\.x, (v\d+) = \2\.y;", ln)
            if mm:
                for h in (0, 1):
                    env[h][mm.group(1)], env[h][mm.group(3)] = env[h][mm.group(2)]
                continue
            mm = re.fullmatch(r"const gar_acc (v\d+) = gar_addbf\(([ly]\d+), (.*)\);", ln)
            if mm:
                for h in (0, 1):
                    env[h][mm.group(1)] = np.float32(env[h][mm.group(2)] + val(h, mm.group(3)))
                continue
            mm = re.fullmatch(r"const gar_acc (v\d+) = gar_op\((.*), (.*)\);", ln)
            if mm:
                for h in (0, 1):
                    env[h][mm.group(1)] = comb(val(h, mm.group(2)), val(h, mm.group(3)))
                continue
            mm = re.fullmatch(r"if \(ok( && !hb)?\) gar_stio\(tout\[(\d+)\] \+ e, (.*)\);", ln)
            if mm:
                for h in ((0,) if mm.group(1) else (0, 1)):
                    v = val(h, mm.group(3))
                    r = (h * m + int(mm.group(2))) % P
                    out[r][e] = _bf16_round(np.float32([v]))[0] if dtype == "bf16" else v
                    written[r][e] += 1
                continue
            raise AssertionError("statement the interpreter does not know: " + ln)
    for r in range(P):
        assert (written[r] == 1).all(), f"rank {r} not written exactly once"
    return out


def _inputs(P, n, dtype, seed):
    rng = np.random.default_rng(seed)
    if dtype == "i32":
        return [rng.integers(-1000, 1000, n).astype(np.int32) for _ in range(P)]
    xs = [(rng.standard_normal(n) * np.exp2(rng.integers(-12, 13, n))).astype(np.float32) for _ in range(P)]
    return [_bf16_round(x) for x in xs] if dtype == "bf16" else xs


def _bits(a, dtype):
    return np.asarray(a).view(np.int32 if dtype == "i32" else np.uint32)


def test_applies_to_latency_optimal_cyclic_only():
    def form(P, S, group="cyclic"):
        old = os.environ.get("GAR_TUNE_FUSED_FORM")
        os.environ["GAR_TUNE_FUSED_FORM"] = "2"
        try:
            return G.gar_plan_get_info(G.gar_plan_create_group(P, 4096, "f32", "sum", S, group))["fused_form"]
        finally:
            if old is None:
                os.environ.pop("GAR_TUNE_FUSED_FORM", None)
            else:
                os.environ["GAR_TUNE_FUSED_FORM"] = old
    assert form(127, 7) == G.GAR_FORM_SPLIT
    assert form(40, 6) == G.GAR_FORM_SPLIT
    assert form(64, 6) == G.GAR_FORM_SPLIT
    assert form(127, 8) == G.GAR_FORM_BREADTH        # K < P: not rotation invariant
    assert form(64, 6, "xor") == G.GAR_FORM_BREADTH


CASES = [(5, "f32", "sum"), (6, "f32", "sum"), (7, "bf16", "sum"), (9, "f32", "max"), (12, "bf16", "sum"),
         (13, "i32", "sum"), (16, "f32", "sum"), (21, "bf16", "sum"), (24, "f32", "min")]


@pytest.mark.parametrize("P,dtype,op", CASES)
def test_generated_code_reproduces_oracle(P, dtype, op):
    """Bit for bit against the oracle for the latency-optimal schedule, n = 2P + 3."""
    n = 2 * P + 3
    xs = _inputs(P, n, dtype, seed=P * 17 + len(dtype))
    S = max(1, (P - 1).bit_length())
    src, info = _split_source(P, n, dtype, S, op)
    assert info["fused_form"] == G.GAR_FORM_SPLIT and info["K"] == P
    got = _run_split(src, P, xs, dtype, op)
    want = O.allreduce(xs, S, op, dtype)
    for x in range(P):
        np.testing.assert_array_equal(_bits(got[x], dtype), _bits(np.asarray(want[x], dtype=got[x].dtype), dtype),
                                      err_msg=f"P={P} rank {x}")


def test_p127_exchange_count():
    """P = 127 latency-optimal: each half evaluates 768 of the 1524 combines (its 64
    placements, one shared with the other half) and receives 126 vectors."""
    src, info = _split_source(127, 4194304, "bf16", 7)
    body = re.search(r"void gar_eval_sp\(.*?\n\}\n", src, re.S).group(0)
    pairs = body.count("__fadd2_rn(make_float2(")
    singles = len(re.findall(r"const gar_acc v\d+ = gar_(?:addbf|op)\(", body))
    assert 2 * pairs + singles == 768
    assert len(re.findall(r"gar_x(?:io|acc)\(hb \?", body)) == 126
    assert body.count("gar_ldio(tin[") == 64 and body.count("gar_stio(tout[") == 64


def test_p127_kernel_reproduces_oracle():
    """The P = 127 latency-optimal two-lane kernel (the shape the GPU sweeps ran),
    interpreted for both halves against the oracle."""
    P, n, S = 127, 6, 7
    xs = _inputs(P, n, "bf16", seed=5)
    src, info = _split_source(P, n, "bf16", S)
    assert info["fused_form"] == G.GAR_FORM_SPLIT
    got = _run_split(src, P, xs, "bf16", "sum")
    want = O.allreduce(xs, S, "sum", "bf16")
    for x in range(P):
        np.testing.assert_array_equal(_bits(got[x], "bf16"), _bits(np.asarray(want[x], dtype=np.float32), "bf16"),
                                      err_msg=f"rank {x}")


def test_interpreter_catches_a_planted_mistake():
    """Swapping the two sources of one exchange breaks the comparison."""
    P, n, S = 7, 17, 3
    xs = _inputs(P, n, "f32", 3)
    src, _ = _split_source(P, n, "f32", S)
    mm = re.search(r"gar_xacc\(hb \? (v\d+) : (v\d+)\)", src)
    bad = src.replace(mm.group(0), f"gar_xacc(hb ? {mm.group(2)} : {mm.group(1)})", 1)
    assert bad != src
    got = _run_split(bad, P, xs, "f32", "sum")
    want = O.allreduce(xs, S, "sum", "f32")
    assert any(not np.array_equal(got[x], want[x]) for x in range(P))


@pytest.mark.parametrize("P", [5, 8, 24, 40, 127])
def test_split_kernels_compile(P):
    old = os.environ.get("GAR_TUNE_FUSED_FORM")
    os.environ["GAR_TUNE_FUSED_FORM"] = "2"
    try:
        S = max(1, (P - 1).bit_length())
        for dtype in ("f32", "bf16", "i32"):
            for op in ("sum", "max"):
                G.gar_plan_compile(G.gar_plan_create(P, 4 * P + 3, dtype, op, S), "fused")
    finally:
        if old is None:
            os.environ.pop("GAR_TUNE_FUSED_FORM", None)
        else:
            os.environ["GAR_TUNE_FUSED_FORM"] = old
