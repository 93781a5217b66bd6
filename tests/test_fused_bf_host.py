"""Host-side checks of the breadth-first fused kernel (no GPU).

The breadth-first form evaluates a plan's combine program step by step, with paired
fp32 adds and bf16 mixed adds.  These tests check, without a GPU:
  * which plans take it (gar_plan_info.fused_form);
  * that its generated evaluation code, run by a small interpreter written here in
    numpy float32, gives the oracle's bits for every rank and element, at every step
    count, for cyclic and XOR groups, sums and max/min, and rotated block layouts;
  * that NVRTC compiles it for sm_103a for a range of plans.
"""

import os
import re

import numpy as np
import pytest

from oracle import gar_oracle as O
from paper_2004_09362_gb300 import gar as G


def _with_form(form, fn):
    old = os.environ.get("GAR_TUNE_FUSED_FORM")
    os.environ["GAR_TUNE_FUSED_FORM"] = str(form)
    try:
        return fn()
    finally:
        if old is None:
            os.environ.pop("GAR_TUNE_FUSED_FORM", None)
        else:
            os.environ["GAR_TUNE_FUSED_FORM"] = old


def _bf_source(P, n, dtype, S, op="sum", group="cyclic"):
    def make():
        pl = G.gar_plan_create_group(P, n, dtype, op, S, group)
        return G.gar_plan_fused_source(pl), G.gar_plan_get_info(pl)
    return _with_form(1, make)


# ---------------------------------------------------------------------------
# Which plans take the breadth-first form
# ---------------------------------------------------------------------------

def test_selection():
    form = {S: G.gar_plan_get_info(G.gar_plan_create(127, 4194304, "bf16", "sum", S))["fused_form"]
            for S in range(7, 15)}
    assert form == {7: 1, 8: 1, 9: 0, 10: 0, 11: 0, 12: 0, 13: 0, 14: 0}
    assert G.gar_plan_get_info(G.gar_plan_create(127, 4096, "f32", "sum", 7))["fused_form"] == 1
    for dtype, op in (("bf16", "max"), ("f32", "min"), ("i32", "sum")):
        assert G.gar_plan_get_info(G.gar_plan_create(127, 4096, dtype, op, 7))["fused_form"] == 0
    for P, S in ((24, 10), (64, 6), (8, 3), (5, 3)):
        assert G.gar_plan_get_info(G.gar_plan_create(P, 4096, "f32", "sum", S))["fused_form"] == 0


def test_every_combine_emitted_once(monkeypatch):
    """P = 127, S = 7 in one pass: the 1524 combines are 2 x (paired adds) + single adds,
    and the even-distance steps pair most of them."""
    monkeypatch.setenv("GAR_TUNE_BF_GROUPS", "1")
    monkeypatch.setenv("GAR_TUNE_BF_WARPS", "1")
    monkeypatch.setenv("GAR_TUNE_BF_MINB", "8")
    src, info = _bf_source(127, 4194304, "bf16", 7)
    body = re.search(r"void gar_eval_bf\(.*?\n\}\n", src, re.S).group(0)
    pairs = body.count("__fadd2_rn(make_float2(")
    singles = len(re.findall(r"const gar_acc v\d+ = gar_(?:addbf|op)\(", body))
    assert 2 * pairs + singles == info["fused_combines"] == 1524
    assert pairs >= 500
    assert "__launch_bounds__(32, 8)" in src      # the shape forced above
    monkeypatch.delenv("GAR_TUNE_BF_WARPS")
    monkeypatch.delenv("GAR_TUNE_BF_MINB")
    src8, _ = _bf_source(127, 4194304, "bf16", 8)
    assert "__launch_bounds__(128, 3)" in src8    # 192 live values: 168 registers


# ---------------------------------------------------------------------------
# Interpreter of the generated evaluation function
# ---------------------------------------------------------------------------

def _bf16_round(x):
    return O.round_to_bf16(np.asarray(x, dtype=np.float32))


def _run_generated(src, P, xs, dtype, op, in_place=False):
    """Evaluates gar_eval_bf for every element e of P rank vectors xs (numpy), returning
    the P output vectors.  The interpreter knows the few statement forms the generator
    emits; rank expressions are evaluated with the element's block b (mod P for the
    doubled pointer tables)."""
    body = re.search(r"void gar_eval_bf\(.*?\{\n(.*?)\n\}\n", src, re.S).group(1)
    n = len(xs[0])
    nblk = re.search(r"return e < big \? \(int\)\(e / (\d+)ULL\) : \(int\)\((\d+)ULL \+ \(e - big\) / (\d+)ULL\)", src)
    bigm = re.search(r"const gar_u64 big = (\d+)ULL;", src)

    def block_of(e):
        if "gar_block_of" not in src:
            return 0
        if nblk is None:
            return e
        q1, rem, q = int(nblk.group(1)), int(nblk.group(2)), int(nblk.group(3))
        big = int(bigm.group(1))
        return e // q1 if e < big else rem + (e - big) // q

    xor = "(b ^" in body

    def rank(expr, b):
        expr = expr.strip()
        val = eval(expr, {}, {"b": b})  # generated arithmetic on b only
        return val % P if not xor else val

    comb = {"sum": lambda a, c: np.float32(a + c), "max": lambda a, c: np.float32(max(a, c)),
            "min": lambda a, c: np.float32(min(a, c))}[op]
    if dtype == "i32":
        comb = {"sum": lambda a, c: np.int32((int(a) + int(c) + 2**31) % 2**32 - 2**31),
                "max": lambda a, c: max(a, c), "min": lambda a, c: min(a, c)}[op]
    out = xs if in_place else [np.zeros_like(x) for x in xs]
    lines = [ln.strip() for ln in body.split("\n") if ln.strip() and not ln.strip().startswith("(void)")]
    N = r"(?:_\d+)?"   # pass suffix of the two-pass form
    for e in range(n):
        b = block_of(e)
        env = {}
        shared = {}

        def val(tok):
            tok = tok.strip()
            m = re.fullmatch(r"gar_wide\((l\d+" + N + r")\)", tok)
            return env[m.group(1)] if m else env[tok]

        for ln in lines:
            if ln.startswith("__shared__ gar_io gar_sl_all[") or ln.startswith("gar_io *const gar_sl = "):
                continue
            m = re.fullmatch(r"gar_sl\[(\d+) \* GAR_BF_THREADS\] = (l\d+);", ln)
            if m:
                shared[int(m.group(1))] = env[m.group(2)]
                continue
            m = re.fullmatch(r"const gar_io (l\d+" + N + r") = gar_sl\[(\d+) \* GAR_BF_THREADS\];", ln)
            if m:
                env[m.group(1)] = shared[int(m.group(2))]
                continue
            m = re.fullmatch(r"const gar_io (l\d+" + N + r") = gar_ldio\((?:a\.in|tin)\[(.*)\] \+ e\);", ln)
            if m:
                env[m.group(1)] = xs[rank(m.group(2), b)][e]
                continue
            m = re.fullmatch(r"const float2 (w\d+" + N + r") = __fadd2_rn\(make_float2\((.*), (.*)\), make_float2\((.*), (.*)\)\);", ln)
            if m:
                env[m.group(1)] = (np.float32(val(m.group(2)) + val(m.group(4))),
                                   np.float32(val(m.group(3)) + val(m.group(5))))
                continue
            m = re.fullmatch(r"const gar_acc (v\d+" + N + r") = (w\d+" + N + r")\.x, (v\d+" + N + r") = \2\.y;", ln)
            if m:
                env[m.group(1)], env[m.group(3)] = env[m.group(2)]
                continue
            m = re.fullmatch(r"const gar_acc (v\d+" + N + r") = gar_addbf\((l\d+" + N + r"), (.*)\);", ln)
            if m:
                env[m.group(1)] = np.float32(env[m.group(2)] + val(m.group(3)))
                continue
            m = re.fullmatch(r"const gar_acc (v\d+" + N + r") = gar_op\((.*), (.*)\);", ln)
            if m:
                env[m.group(1)] = comb(val(m.group(2)), val(m.group(3)))
                continue
            m = re.fullmatch(r"gar_stio\((?:a\.out|tout)\[(.*)\] \+ e, (.*)\);", ln)
            if m:
                v = val(m.group(2))
                out[rank(m.group(1), b)][e] = _bf16_round(np.float32([v]))[0] if dtype == "bf16" else v
                continue
            raise AssertionError("statement the interpreter does not know: " + ln)
    return out


def _inputs(P, n, dtype, seed):
    rng = np.random.default_rng(seed)
    if dtype == "i32":
        return [rng.integers(-1000, 1000, n).astype(np.int32) for _ in range(P)]
    xs = [(rng.standard_normal(n) * np.exp2(rng.integers(-12, 13, n))).astype(np.float32) for _ in range(P)]
    return [_bf16_round(x) for x in xs] if dtype == "bf16" else xs


CASES = ([(P, "f32", "sum", "cyclic") for P in (3, 5, 6, 7, 9, 12, 13)] +
         [(7, "bf16", "sum", "cyclic"), (11, "bf16", "sum", "cyclic"), (6, "f32", "max", "cyclic"),
          (5, "i32", "min", "cyclic"), (8, "f32", "sum", "xor"), (16, "bf16", "sum", "xor")])


@pytest.mark.parametrize("P,dtype,op,group", CASES)
def test_generated_code_reproduces_oracle(P, dtype, op, group):
    """Bit for bit against the oracle at every step count in [L, 2L] with more than one
    result copy, with n = 3P + 2 (ragged blocks, every rotation b)."""
    n = 3 * P + 2
    xs = _inputs(P, n, dtype, seed=P * 31 + len(dtype))
    L = max(1, (P - 1).bit_length())
    for S in range(L, 2 * L):
        src, info = _bf_source(P, n, dtype, S, op, group)
        assert info["K"] > 1
        got = _run_generated(src, P, xs, dtype, op)
        want = O.allreduce(xs, S, op, dtype, group=group)
        for x in range(P):
            np.testing.assert_array_equal(np.asarray(got[x]).view(np.uint32 if dtype != "i32" else np.int32),
                                          np.asarray(want[x], dtype=got[x].dtype).view(np.uint32 if dtype != "i32" else np.int32),
                                          err_msg=f"P={P} S={S} rank {x}")


@pytest.mark.parametrize("groups", [2, 3])
@pytest.mark.parametrize("P,dtype,op,group", [(5, "f32", "sum", "cyclic"), (7, "bf16", "sum", "cyclic"),
                                              (12, "f32", "sum", "cyclic"), (13, "bf16", "sum", "cyclic"),
                                              (6, "f32", "max", "cyclic"), (8, "f32", "sum", "xor")])
def test_generated_passes_reproduce_oracle(P, dtype, op, group, groups, monkeypatch):
    """The form evaluated in several passes over placement groups (the default for the
    widest programs, forced here on small ones): bit for bit against the oracle at every
    step count with several result copies, ragged blocks.  The in-place Allreduce
    overwrites contributions with results during the first pass, so later passes must
    take the contributions from the shared-memory copy; the interpreter writes the
    results into the same arrays it reads the contributions from, as the kernel does."""
    monkeypatch.setenv("GAR_TUNE_BF_GROUPS", str(groups))
    n = 3 * P + 2
    xs = _inputs(P, n, dtype, seed=P * 7 + groups)
    L = max(1, (P - 1).bit_length())
    for S in range(L, 2 * L):
        src, info = _bf_source(P, n, dtype, S, op, group)
        assert "gar_sl[" in src
        got = _run_generated(src, P, [x.copy() for x in xs], dtype, op, in_place=True)
        want = O.allreduce(xs, S, op, dtype, group=group)
        for x in range(P):
            np.testing.assert_array_equal(np.asarray(got[x]).view(np.uint32 if dtype != "i32" else np.int32),
                                          np.asarray(want[x], dtype=got[x].dtype).view(np.uint32 if dtype != "i32" else np.int32),
                                          err_msg=f"P={P} S={S} groups={groups} rank {x}")


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_p127_latency_optimal_kernel_reproduces_oracle(dtype):
    """The kernel text the P = 127 latency-optimal plan runs by default (breadth-first,
    two passes; it does not depend on n for an unrotated program, so a 6-element plan
    has the same text as the 8 MiB one), interpreted in place against the oracle."""
    P, n, S = 127, 6, 7
    xs = _inputs(P, n, dtype, seed=11)
    src = G.gar_plan_fused_source(G.gar_plan_create(P, n, dtype, "sum", S))
    assert src == G.gar_plan_fused_source(G.gar_plan_create(P, 4194304, dtype, "sum", S))
    assert "gar_sl[" in src
    got = _run_generated(src, P, [x.copy() for x in xs], dtype, "sum", in_place=True)
    want = O.allreduce(xs, S, "sum", dtype)
    for x in range(P):
        np.testing.assert_array_equal(np.asarray(got[x]).view(np.uint32),
                                      np.asarray(want[x], dtype=np.float32).view(np.uint32), err_msg=f"rank {x}")


def test_interpreter_catches_a_pass_reading_overwritten_contributions(monkeypatch):
    """Planted mistake: later passes reading the contributions from global memory, where
    the first pass has already stored results in place, break the comparison."""
    monkeypatch.setenv("GAR_TUNE_BF_GROUPS", "2")
    P, n, S = 7, 23, 3
    xs = _inputs(P, n, "f32", 5)
    src, _ = _bf_source(P, n, "f32", S)
    bad = re.sub(r"const gar_io (l\d+_\d+) = gar_sl\[(\d+) \* GAR_BF_THREADS\];",
                 lambda m: f"const gar_io {m.group(1)} = gar_ldio(a.in[{m.group(2)}] + e);", src)
    assert bad != src
    got = _run_generated(bad, P, [x.copy() for x in xs], "f32", "sum", in_place=True)
    want = O.allreduce(xs, S, "sum", "f32")
    assert any(not np.array_equal(got[x], want[x]) for x in range(P))


def test_two_passes_for_the_widest_programs():
    """P = 127, S = 7 evaluates its results in two passes (1752 combines: the shared
    values are computed again) in 128-thread CTAs; S = 8 in one."""
    src, info = _bf_source(127, 4194304, "bf16", 7)
    body = re.search(r"void gar_eval_bf\(.*?\n\}\n", src, re.S).group(0)
    pairs = body.count("__fadd2_rn(make_float2(")
    singles = len(re.findall(r"const gar_acc v\d+(?:_\d+)? = gar_(?:addbf|op)\(", body))
    assert 2 * pairs + singles == 1752
    assert body.count("gar_ldio(") == 127 and body.count("gar_stio(") == 127
    assert "__launch_bounds__(128, 3)" in src
    src8, _ = _bf_source(127, 4194304, "bf16", 8)
    assert "gar_sl[" not in src8


def test_interpreter_catches_a_planted_mistake():
    """The interpreter is not vacuous: swapping two result stores in the generated text
    breaks the comparison."""
    P, n, S = 7, 23, 3
    xs = _inputs(P, n, "f32", 5)
    src, _ = _bf_source(P, n, "f32", S)
    stores = re.findall(r"gar_stio\(a\.out\[(\d+)\] \+ e, (v\d+)\);", src)
    (r0, v0), (r1, v1) = stores[0], stores[1]
    bad = src.replace(f"a.out[{r0}] + e, {v0});", "@@").replace(f"a.out[{r1}] + e, {v1});", f"a.out[{r1}] + e, {v0});")
    bad = bad.replace("@@", f"a.out[{r0}] + e, {v1});")
    assert bad != src
    got = _run_generated(bad, P, xs, "f32", "sum")
    want = O.allreduce(xs, S, "sum", "f32")
    assert any(not np.array_equal(got[x], want[x]) for x in range(P))


# ---------------------------------------------------------------------------
# NVRTC compiles the form (host only)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("P", [2, 3, 5, 8, 12, 24, 33])
def test_breadth_first_kernels_compile(P):
    def go():
        L = max(1, (P - 1).bit_length())
        for dtype in ("f32", "bf16", "i32"):
            for op in ("sum", "max"):
                for S in range(L, 2 * L + 1):
                    G.gar_plan_compile(G.gar_plan_create(P, 4 * P + 3, dtype, op, S), "fused")
        if P & (P - 1) == 0:
            G.gar_plan_compile(G.gar_plan_create_group(P, 1000, "f32", "sum", L, "xor"), "fused")
    _with_form(1, go)



@pytest.mark.parametrize("groups", [2, 3])
def test_pass_kernels_compile(groups, monkeypatch):
    """NVRTC compiles the several-pass form (shared-memory copy of the contributions,
    suffixed values) for rotated and unrotated programs, sums and max."""
    monkeypatch.setenv("GAR_TUNE_FUSED_FORM", "1")
    monkeypatch.setenv("GAR_TUNE_BF_GROUPS", str(groups))
    for P in (5, 12, 33):
        L = max(1, (P - 1).bit_length())
        for dtype in ("f32", "bf16"):
            for op in ("sum", "max"):
                for S in (L, L + 1):
                    G.gar_plan_compile(G.gar_plan_create(P, 4 * P + 3, dtype, op, S), "fused")


def test_default_p127_latency_optimal_kernel_compiles():
    """The P = 127 latency-optimal default (two passes) compiles for sm_103a."""
    G.gar_plan_compile(G.gar_plan_create(127, 4096, "bf16", "sum", 7), "fused")


def test_fused_form_matches_generated_kernel():
    """gar_plan_info.fused_form names the kernel the plan's source defines."""
    for P in (5, 24, 64, 127):
        L = max(1, (P - 1).bit_length())
        for S in range(L, 2 * L + 1):
            pl = G.gar_plan_create(P, 4096, "bf16", "sum", S)
            form = G.gar_plan_get_info(pl)["fused_form"]
            src = G.gar_plan_fused_source(pl)
            assert ("gar_fusedbf_" in src) == (form == G.GAR_FORM_BREADTH), (P, S)
            assert ("gar_fused_P" in src) == (form == G.GAR_FORM_SINGLE), (P, S)
