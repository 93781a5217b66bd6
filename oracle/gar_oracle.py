"""Plain, slow CPU oracle: P simulated processes running the paper's Allreduce.

TEST INFRASTRUCTURE, NOT PRODUCT CODE (see ``oracle/__init__.py``).

Source: D. Kolmakov, X. Zhang, "A Generalization of the Allreduce Operation",
arXiv 2004.09362.  Section and equation labels below are the paper's own.

Model (Sec. "Communication description via permutations")
----------------------------------------------------------
* P processes 0..P-1.  Process j owns the vector V_j = (u_{0,j}, ..., u_{P-1,j}) of P
  blocks (eq. initial_data).  Blocks are unequal when P does not divide n (the paper
  assumes u = m/P, Sec. "Communication model"); we use the MPI reduce_scatter split:
  the first n mod P blocks get one extra element (reading C3).
* T_P is the cyclic group t_k(x) = x + k mod P with generator c = (0 1 ... P-1)
  (Table 1a); the placement permutation h is the identity (eq. distr_vector_def,
  reading C4).
* A distributed vector t_k q has its block i on process t_k(h(i)) = i + k (eq.
  distr_vector).  Its *content* says where each block's terms come from: the initial
  vector t_k q_k holds u_{i,i+k} in block i, so a leaf "k" means "block i comes from
  process i + k".  Combining two same-placement vectors (eq.
  distr_vectors_combination) makes a node (own, received).
* A communication operator t_l moves every block from process x to process x + l
  (eq. comm_op_0).  All processes send and receive at once.

Schedule (Secs. "Bandwidth-optimal algorithm", "Moving towards latency-optimal
version", "Latency-optimal version")
----------------------------------------------------------------------
* N_0 = P, N_{i+1} = ceil(N_i / 2) (eq. bo_starting_set_size); L = ceil(log2 P) steps
  bring N to 1.
* Reduction step i: the vectors with index k in [ceil(N_i/2), N_i - 1] (eq.
  bo_tx_dist) are moved by t^{-floor(N_i/2)} (eq. bo_dir_perms) and each is combined
  with the vector that now shares its placement (eqs. bo_step_even, bo_step_odd); when
  N_i is odd the vector with index 0 (q*) sits the step out.
* To remove r distribution steps, the reduction phase runs K copies of that schedule,
  copy s shifted by s (vector indices +s, same operators; eq. var_starting_set and the
  equations after it), so that it ends with q_Sigma at placements 0..K-1.  Vectors of
  different copies that have the same placement and the same content are the same
  vector and are sent and combined once.  q* and q' vectors are never merged even at
  equal placement (Sec. "Latency-optimal version").  The paper says "double the number
  of resulting vectors" (2^r); the smallest K that lets the remaining distribution
  steps finish is K = N_{L-r}, which equals 2^r when P is a power of two (reading C7).
  r = L (K = P) is the latency-optimal version; r = 0 (K = 1) the bandwidth-optimal one.
* Distribution phase: the reduction steps i = L-r-1, ..., 0 in reverse, with no
  combination: the vectors at placements [N_i mod 2, ceil(N_i/2) - 1] are copied by
  t^{+floor(N_i/2)} (end of Sec. "Bandwidth-optimal algorithm").
* Result: process x's block b is the vector at placement (x - b) mod P.

Groups: T_P is the cyclic group (Table 1a) by default.  group="xor" uses the
self-inverse group of Table 1b (t_k(x) = x XOR k, P a power of two).  Everything above
is written with the group operation: placement k puts block i on process t_k(i); a step
moves the transmitted vectors by the group element that takes index k to index
k - floor(N_i/2), which is t_{floor(N_i/2)}^{-1} (t^{-floor(N_i/2)} in the cyclic group,
t_{N_i/2} itself in the XOR group, where k - N_i/2 = k XOR N_i/2 for the transmitted
indices); copy s of the schedule has index k at placement t_s(k); distribution moves by
t_{floor(N_i/2)} (reading C18).

Precision: f32 runs in float32 (IEEE round-to-nearest-even, as numpy does it); i32 in
int32 with two's-complement wraparound; bf16 inputs are widened exactly to float32,
every partial is float32, and each q_Sigma is rounded to bf16 once, at the end of the
reduction phase (reading C6).  max/min are exact in every type.

Message sizes: a message element counts the size of the type it travels in: a leaf
(an input block, not yet combined) travels in the input type, a combined partial in the
accumulation type (float32 for bf16), a distribution-phase block in the output type.
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

__all__ = [
    "OPS", "DTYPES", "ceil_log2", "vector_counts", "block_bounds", "schedule_shape",
    "ExprTable", "Run", "simulate", "allreduce", "round_to_bf16", "is_bf16_exact",
    "column_reduce_exact", "kahan_sum_f64", "tree_string", "parse_tree",
    "eval_tree", "cost_model_time", "optimal_steps", "group_ops", "simulate_ring",
    "fold_sequence",
]

OPS = ("sum", "max", "min")
DTYPES = ("f32", "bf16", "i32")
_ITEMSIZE = {"f32": 4, "bf16": 2, "i32": 4}
_ACC_ITEMSIZE = {"f32": 4, "bf16": 4, "i32": 4}


# ---------------------------------------------------------------------------
# Schedule arithmetic
# ---------------------------------------------------------------------------

def ceil_log2(P: int) -> int:
    """L = ceil(log2 P): the number of reduction steps (Sec. "Bandwidth-optimal
    algorithm": the reduction phase takes ceil(log P) steps).

    Pinned by: test_step_counts.
    """
    if P < 1:
        raise ValueError("P must be >= 1")
    L = 0
    while (1 << L) < P:
        L += 1
    return L


def vector_counts(P: int) -> list[int]:
    """[N_0, ..., N_L] with N_0 = P and N_{i+1} = ceil(N_i / 2) (eq.
    bo_starting_set_size).

    Pinned by: test_step_counts, test_planted_floor_halving_is_caught.
    """
    Ns = [P]
    while Ns[-1] > 1:
        Ns.append((Ns[-1] + 1) // 2)
    return Ns


def block_bounds(n: int, P: int) -> list[tuple[int, int]]:
    """Block i of every vector (eq. initial_data).  The paper assumes equal blocks
    u = m/P (Sec. "Communication model"); for P not dividing n the first n mod P blocks
    get one extra element (reading C3).

    Pinned by: test_block_bounds_reading_c3 (hand-written sizes),
    test_planted_partition_mistake_is_caught.
    """
    q, rem = divmod(n, P)
    out, start = [], 0
    for i in range(P):
        size = q + (1 if i < rem else 0)
        out.append((start, start + size))
        start += size
    assert start == n
    return out


def schedule_shape(P: int, steps: int) -> dict:
    """Step count S in [L, 2L] (abstract; Sec. "Moving towards latency-optimal
    version": S = 2 ceil(log P) - r, 0 <= r <= ceil(log P)).  Returns L, S, r and the
    number K of q_Sigma copies the reduction phase must end with (reading C7:
    K = N_{L-r}).  Even S in (2L, 2(P-1)] selects the fold schedule (fold_sequence;
    K = 1), the step counts toward the Ring that Sec. "Conclusion" leaves to future work
    (reading C19).

    Pinned by: test_step_counts, test_fold_schedule.
    """
    L = ceil_log2(P)
    if L <= steps <= 2 * L:
        r = 2 * L - steps
        K = vector_counts(P)[L - r]
        return {"P": P, "L": L, "S": steps, "r": r, "K": K}
    if steps > 2 * L and steps <= 2 * (P - 1) and steps % 2 == 0:
        return {"P": P, "L": L, "S": steps, "r": 0, "K": 1}
    raise ValueError(f"steps={steps} outside [{L}, {2 * L}] and not an even count up to "
                     f"{2 * (P - 1)} for P={P}")


def fold_sequence(P: int, F: int) -> list[int]:
    """Vectors folded per reduction step for F steps (reading C19).  A step with N
    vectors and fold f moves the vectors with index [N-f, N) by t^{-f} onto [N-2f, N-f)
    and combines them there; f = floor(N/2) is the bandwidth-optimal step (eqs.
    bo_tx_dist, bo_dir_perms), f = 1 moves one vector by the generator.  F = L gives the
    bandwidth-optimal halving; F > L spreads the P-1 folds as evenly as the constraints
    allow (1 <= f <= floor(N/2), and the remaining steps must still reach N = 1).

    Pinned by: test_fold_schedule, test_fold_schedule_ends.
    """
    L = ceil_log2(P)
    if not (L <= F <= max(P - 1, L)):
        raise ValueError("F out of range")
    if F == L:
        Ns = vector_counts(P)
        return [N // 2 for N in Ns[:-1]]
    folds, N = [], P
    for i in range(F):
        r = F - i
        lo = max(1, N - 2 ** (r - 1))
        hi = min(N // 2, N - r)
        want = -(-(N - 1) // r)          # ceil((N-1)/r): an even share of what is left
        f = min(max(want, lo), hi)
        folds.append(f)
        N -= f
    assert N == 1
    return folds


# ---------------------------------------------------------------------------
# Contents of distributed vectors (symbolic)
# ---------------------------------------------------------------------------

class ExprTable:
    """Interned contents.  A leaf k is the initial vector t_k q_k (block i from process
    i + k, eq. initial_distr_vector); a pair (a, b) is the combination "own (+)
    received" of two same-placement vectors (eq. distr_vectors_combination).

    Pinned by: test_golden_tree (hand-derived trees),
    test_every_output_covers_every_rank_once.
    """

    def __init__(self):
        self.nodes: list = []          # id -> ("leaf", k) | ("pair", a, b)
        self._leaf: dict[int, int] = {}
        self._pair: dict[tuple[int, int], int] = {}

    def leaf(self, k: int) -> int:
        if k not in self._leaf:
            self._leaf[k] = len(self.nodes)
            self.nodes.append(("leaf", k))
        return self._leaf[k]

    def pair(self, a: int, b: int) -> int:
        key = (a, b)
        if key not in self._pair:
            self._pair[key] = len(self.nodes)
            self.nodes.append(("pair", a, b))
        return self._pair[key]

    def is_leaf(self, e: int) -> bool:
        return self.nodes[e][0] == "leaf"

    def tree(self, e: int):
        """Nested tuples of leaf offsets."""
        node = self.nodes[e]
        if node[0] == "leaf":
            return node[1]
        return (self.tree(node[1]), self.tree(node[2]))

    def leaves(self, e: int) -> list[int]:
        out, stack = [], [e]
        while stack:
            node = self.nodes[stack.pop()]
            if node[0] == "leaf":
                out.append(node[1])
            else:
                stack.append(node[2])
                stack.append(node[1])
        return out


def tree_string(t) -> str:
    """'(a+b)' notation for a nested-tuple tree; leaves are integers.

    Pinned by: test_tree_notation_round_trip.
    """
    if isinstance(t, int):
        return str(t)
    return "(" + tree_string(t[0]) + "+" + tree_string(t[1]) + ")"


def parse_tree(s: str):
    """Inverse of tree_string (used for the hand-derived fixtures in tests/golden).

    Pinned by: test_tree_notation_round_trip.
    """
    s = s.replace(" ", "")
    pos = 0

    def node():
        nonlocal pos
        if s[pos] == "(":
            pos += 1
            a = node()
            assert s[pos] == "+", s
            pos += 1
            b = node()
            assert s[pos] == ")", s
            pos += 1
            return (a, b)
        start = pos
        while pos < len(s) and s[pos].isdigit():
            pos += 1
        return int(s[start:pos])

    t = node()
    assert pos == len(s), s
    return t


def eval_tree(t, leaf_value, op: str):
    """Evaluate a nested-tuple tree with leaf_value(k) at the leaves, combining with op
    in whatever numpy type the leaves carry.

    Pinned by: test_golden_tree_values.
    """
    if isinstance(t, int):
        return leaf_value(t)
    return _combine(op, eval_tree(t[0], leaf_value, op), eval_tree(t[1], leaf_value, op))


def group_ops(P: int, group: str):
    """(op, inverse) of the permutation group T_P acting on {0..P-1}: t_a(t_b(x)) =
    op(op(x, b), a).  "cyclic": t_k(x) = x + k mod P (Table 1a); "xor": t_k(x) = x XOR k,
    the self-inverse group generated by the h_i of Table 1b (P a power of two).

    Pinned by: test_xor_group_bo_is_recursive_halving,
    test_xor_group_lo_is_recursive_doubling.
    """
    if group == "cyclic":
        return (lambda a, b: (a + b) % P), (lambda a: (-a) % P)
    if group == "xor":
        if P & (P - 1):
            raise ValueError("the XOR group (Table 1b) needs P a power of two")
        return (lambda a, b: a ^ b), (lambda a: a)
    raise ValueError(group)


def _reduce_partner(x: int, d: int, P: int, group: str = "cyclic") -> int:
    """Where process x sends during a reduction step: the step operator
    t_d^{-1} (t^{-d} in the cyclic group, eqs. comm_op_0, bo_dir_perms) moves every
    block from x to t_d^{-1}(x).

    Pinned by: test_tx_sets_and_partners, test_planted_wrong_partner_is_caught.
    """
    op, inv = group_ops(P, group)
    return op(x, inv(d))


def _distribute_partner(x: int, d: int, P: int, group: str = "cyclic") -> int:
    """Where process x sends during a distribution step: the reversed operator t_d
    (t^{+d} in the cyclic group; end of Sec. "Bandwidth-optimal algorithm").

    Pinned by: test_int32_bruteforce, test_ring_equals_textbook_ring.
    """
    op, _inv = group_ops(P, group)
    return op(x, d)


def _combine(op: str, a, b):
    """The reduction operator (+) of the Allreduce (Sec. "Combination of distributed
    data vectors"); elementwise, in the operands' own numpy type.

    Pinned by: test_int32_bruteforce, test_planted_sign_error_is_caught.
    """
    if op == "sum":
        return a + b
    if op == "max":
        return np.maximum(a, b)
    if op == "min":
        return np.minimum(a, b)
    raise ValueError(op)


# ---------------------------------------------------------------------------
# bf16 rounding (reading C6), written from the format's definition
# ---------------------------------------------------------------------------

def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even), returned as float32.
    bfloat16 keeps the top 16 bits of the float32 encoding (sign, 8 exponent bits,
    7 fraction bits); rounding looks at the 16 discarded bits.  Finite inputs only.

    Pinned by: test_bf16_rounding_matches_library (torch's conversion).
    """
    x = np.ascontiguousarray(x, dtype=np.float32)
    bits = x.view(np.uint32).astype(np.uint64)
    upper = bits >> np.uint64(16)
    lower = bits & np.uint64(0xFFFF)
    half = np.uint64(0x8000)
    round_up = (lower > half) | ((lower == half) & ((upper & np.uint64(1)) == np.uint64(1)))
    upper = upper + round_up.astype(np.uint64)
    out = (upper << np.uint64(16)).astype(np.uint32)
    return out.view(np.float32)


def is_bf16_exact(x: np.ndarray) -> bool:
    x = np.ascontiguousarray(x, dtype=np.float32)
    return bool(np.all((x.view(np.uint32) & np.uint32(0xFFFF)) == 0))


# ---------------------------------------------------------------------------
# The simulation
# ---------------------------------------------------------------------------

@dataclass
class Run:
    """Everything one simulated Allreduce produced.

    Pinned by: test_is_bf16_exact.
    """
    P: int
    n: int
    steps: int
    L: int
    r: int
    K: int
    op: str
    dtype: str
    exprs: ExprTable
    outputs: list | None                 # per rank: array over the selected elements
    out_key: list = field(default_factory=list)   # out_key[x][b] = (placement, expr)
    log: list = field(default_factory=list)       # one dict per communication step
    after_reduction: list = field(default_factory=list)  # per shift s: key at placement s
    states: list = field(default_factory=list)    # per reduction step: per shift: keys
    combines: list = field(default_factory=list)  # per reduction step: distinct combines

    def output_tree(self, x: int, b: int):
        return self.exprs.tree(self.out_key[x][b][1])

    def message_elems_per_rank(self, x: int) -> int:
        """Elements rank x sends over the whole Allreduce."""
        tot = 0
        for st in self.log:
            for (src, _dst, items) in st["messages"]:
                if src == x:
                    tot += sum(cnt for (_k, cnt, _sz) in items)
        return tot

    def message_blocks_per_rank(self, x: int) -> int:
        tot = 0
        for st in self.log:
            for (src, _dst, items) in st["messages"]:
                if src == x:
                    tot += len(items)
        return tot

    def step_bytes(self) -> list[int]:
        """Bytes sent per communication step, summed over all processes."""
        return [sum(cnt * sz for (_s, _d, items) in st["messages"] for (_k, cnt, sz) in items)
                for st in self.log]


def simulate(P: int, n: int, steps: int, inputs=None, op: str = "sum",
             dtype: str = "f32", elements=None, group: str = "cyclic") -> Run:
    """Run the Allreduce schedule with P explicit process stores and explicit
    per-step message lists.

    inputs: None for a symbolic run (contents and messages only), else a sequence of P
      1-D numpy arrays of length n (float32 for f32/bf16 -- bf16 values must be exactly
      representable -- or int32 for i32).
    elements: optional sorted array of global element indices; the run then carries
      only those elements (every operation is elementwise, so they come out exactly as
      in a full run).  Message sizes are always those of the full vectors.

    Pinned by: every test in tests/test_oracle_pins.py.
    """
    if op not in OPS:
        raise ValueError(op)
    if dtype not in DTYPES:
        raise ValueError(dtype)
    gop, ginv = group_ops(P, group)
    shape = schedule_shape(P, steps)
    if group == "xor" and steps > 2 * ceil_log2(P):
        raise ValueError("fold schedules beyond 2L use the cyclic group")
    L, r, K = shape["L"], shape["r"], shape["K"]
    if steps > 2 * L:                       # fold schedule (reading C19)
        folds = fold_sequence(P, steps // 2)
    else:
        folds = [N // 2 for N in vector_counts(P)[:-1]]
    Ns = [P]
    for f in folds:
        Ns.append(Ns[-1] - f)
    R = len(folds)                          # reduction steps
    bounds = block_bounds(n, P)
    block_len = [hi - lo for (lo, hi) in bounds]
    ex = ExprTable()
    itemsize = _ITEMSIZE[dtype]
    acc_itemsize = _ACC_ITEMSIZE[dtype]

    # Per-block element selection (global indices inside the block).
    if elements is None:
        sel = [np.arange(lo, hi, dtype=np.int64) for (lo, hi) in bounds]
    else:
        elements = np.asarray(elements, dtype=np.int64)
        sel = [elements[(elements >= lo) & (elements < hi)] for (lo, hi) in bounds]

    have_values = inputs is not None
    if have_values:
        if len(inputs) != P:
            raise ValueError("need one input vector per process")
        want = np.int32 if dtype == "i32" else np.float32
        inputs = [np.asarray(v) for v in inputs]
        for v in inputs:
            if v.shape != (n,) or v.dtype != want:
                raise ValueError(f"input must be shape ({n},) {want}")
            if dtype == "bf16" and not is_bf16_exact(v):
                raise ValueError("bf16 inputs must be exactly representable in bf16")

    # --- initial data: Q_initial = t_0 q_0 : t_1 q_1 : ... : t_{P-1} q_{P-1}
    # (eq. distr_vector_set).  Process x holds block b = t_k^{-1}(x) of t_k q_k (block b
    # sits on t_k(b) = x), which is its own block u_{b, x}.
    store = [dict() for _ in range(P)]
    for x in range(P):
        for k in range(P):
            key = (k, ex.leaf(k))
            b = gop(x, ginv(k))
            store[x][key] = inputs[x][sel[b]].copy() if have_values else None

    # Each shifted copy s of the schedule starts from the same initial set, its index k
    # naming the vector at placement t_s(k) (s + k in the cyclic group; eq.
    # var_starting_set).
    sched = [[(gop(s, k), ex.leaf(gop(s, k))) for k in range(P)] for s in range(K)]
    run = Run(P=P, n=n, steps=steps, L=L, r=r, K=K, op=op, dtype=dtype, exprs=ex,
              outputs=None)

    # --- reduction phase: R steps (L for S in [L, 2L])
    for i in range(R):
        N = Ns[i]
        d = folds[i]          # operator t^{-floor(N_i/2)} (eq. bo_dir_perms); t^{-f} for folds
        c = N - d             # first transmitted index: ceil(N_i/2) when d = floor(N_i/2)
        # Q_TX,i of every shifted copy (eq. bo_tx_dist and its shifted form), each
        # distinct (placement, content) vector once.
        tx = []
        seen = set()
        for s in range(K):
            for k in range(c, N):
                key = sched[s][k]
                if key not in seen:
                    seen.add(key)
                    tx.append(key)
        # Communication: process x sends its blocks of the TX vectors to x - d.
        messages = []
        inbox = [dict() for _ in range(P)]
        for x in range(P):
            dst = _reduce_partner(x, d, P, group)
            items = []
            for key in tx:
                b = gop(x, ginv(key[0]))
                sz = itemsize if ex.is_leaf(key[1]) else acc_itemsize
                items.append((key, block_len[b], sz))
                # the block keeps its index; its placement moves by t_d^{-1}
                moved = (gop(key[0], ginv(d)), key[1])
                inbox[dst][moved] = store[x][key]
            messages.append((x, dst, items))
        run.log.append({"phase": "reduce", "i": i, "N": N, "d": d,
                        "tx": list(tx), "messages": messages})
        # Combination (eqs. bo_step_even / bo_step_odd and their shifted forms).
        new_store = [dict() for _ in range(P)]
        new_sched = []
        step_combines = []
        combined = set()
        for s in range(K):
            q = sched[s]
            nq = []
            for k in range(c):
                if k < N - 2 * d:
                    key = q[k]                 # sits this step out (q* when N is odd)
                    for x in range(P):
                        new_store[x][key] = store[x][key]
                else:
                    own = q[k]
                    moved = (gop(q[k + d][0], ginv(d)), q[k + d][1])
                    assert moved[0] == own[0]
                    key = (own[0], ex.pair(own[1], moved[1]))
                    if key not in combined:
                        combined.add(key)
                        step_combines.append(key)
                        for x in range(P):
                            if have_values:
                                new_store[x][key] = _combine(op, store[x][own], inbox[x][moved])
                            else:
                                new_store[x][key] = None
                nq.append(key)
            new_sched.append(nq)
        sched = new_sched
        store = new_store
        run.states.append([list(q) for q in sched])
        run.combines.append(step_combines)

    # --- end of the reduction phase: shift s holds q_Sigma at placement s
    for s in range(K):
        assert len(sched[s]) == 1 and sched[s][0][0] == s
    run.after_reduction = [sched[s][0] for s in range(K)]
    at_place = {s: sched[s][0] for s in range(K)}
    if have_values and dtype == "bf16":
        # one rounding of each result to bf16 (reading C6)
        for x in range(P):
            for s in range(K):
                key = at_place[s]
                store[x][key] = round_to_bf16(store[x][key])

    # --- distribution phase: reduction steps R-r-1 .. 0 reversed, no combination
    for i in range(R - r - 1, -1, -1):
        N = Ns[i]
        d = folds[i]
        c = N - d
        senders = list(range(N - 2 * d, c))
        messages = []
        inbox = [dict() for _ in range(P)]
        for x in range(P):
            dst = _distribute_partner(x, d, P, group)
            items = []
            for p in senders:
                key = at_place[p]
                b = gop(x, ginv(p))
                items.append((key, block_len[b], itemsize))
                inbox[dst][(gop(p, d), key[1])] = store[x][key]
            messages.append((x, dst, items))
        run.log.append({"phase": "distribute", "i": i, "N": N, "d": d,
                        "tx": [at_place[p] for p in senders], "messages": messages})
        for p in senders:
            newkey = (gop(p, d), at_place[p][1])
            assert gop(p, d) not in at_place
            at_place[gop(p, d)] = newkey
            for x in range(P):
                store[x][newkey] = inbox[x][newkey]

    assert sorted(at_place) == list(range(P))

    # --- result: process x's block b sits at the placement p with t_p(b) = x
    run.out_key = [[at_place[gop(x, ginv(b))] for b in range(P)] for x in range(P)]
    if have_values:
        outs = []
        for x in range(P):
            parts = [store[x][run.out_key[x][b]] for b in range(P)]
            outs.append(np.concatenate(parts) if parts else np.zeros(0, inputs[x].dtype))
        run.outputs = outs
    return run


def simulate_ring(P: int, n: int, inputs=None, op: str = "sum", dtype: str = "f32",
                  elements=None) -> Run:
    """The Ring algorithm: the straightforward Allreduce of Sec. "Allreduce as
    permutation composition" with the cyclic group, whose operator t_{i->0} reduces to the
    generator t (x -> x + 1).  Reduction step i (i = 0..P-2): the partial vector at
    placement i moves by t to placement i + 1 and is combined with the initial vector
    t^{i+1} q_{i+1} there (eq. ring_reduce: own t^{i+1} q_{i+1} (+) received).  After P-1
    steps placement P-1 holds q_Sigma; the distribution phase moves copies by t again,
    P-1 more steps (2(P-1) in total, eq. naive_cost).

    Pinned by: test_ring_equals_textbook_ring, test_ring_steps_traffic_and_tree.
    """
    if op not in OPS:
        raise ValueError(op)
    if dtype not in DTYPES:
        raise ValueError(dtype)
    bounds = block_bounds(n, P)
    block_len = [hi - lo for (lo, hi) in bounds]
    ex = ExprTable()
    itemsize, acc_itemsize = _ITEMSIZE[dtype], _ACC_ITEMSIZE[dtype]
    if elements is None:
        sel = [np.arange(lo, hi, dtype=np.int64) for (lo, hi) in bounds]
    else:
        elements = np.asarray(elements, dtype=np.int64)
        sel = [elements[(elements >= lo) & (elements < hi)] for (lo, hi) in bounds]
    have_values = inputs is not None
    if have_values:
        want = np.int32 if dtype == "i32" else np.float32
        inputs = [np.asarray(v) for v in inputs]
        for v in inputs:
            if v.shape != (n,) or v.dtype != want:
                raise ValueError(f"input must be shape ({n},) {want}")
            if dtype == "bf16" and not is_bf16_exact(v):
                raise ValueError("bf16 inputs must be exactly representable in bf16")
    L = ceil_log2(P)
    run = Run(P=P, n=n, steps=2 * (P - 1), L=L, r=0, K=1, op=op, dtype=dtype, exprs=ex,
              outputs=None)
    store = [dict() for _ in range(P)]
    for x in range(P):
        for k in range(P):
            b = (x - k) % P
            store[x][(k, ex.leaf(k))] = inputs[x][sel[b]].copy() if have_values else None
    cur = (0, ex.leaf(0)) if P > 0 else None      # the partial q', at placement 0
    for i in range(P - 1):
        messages, inbox = [], [dict() for _ in range(P)]
        for x in range(P):
            dst = (x + 1) % P                      # operator t
            b = (x - cur[0]) % P
            sz = itemsize if ex.is_leaf(cur[1]) else acc_itemsize
            messages.append((x, dst, [(cur, block_len[b], sz)]))
            inbox[dst][((cur[0] + 1) % P, cur[1])] = store[x][cur]
        run.log.append({"phase": "reduce", "i": i, "N": None, "d": -1, "tx": [cur],
                        "messages": messages})
        own = ((i + 1) % P, ex.leaf((i + 1) % P))
        key = (own[0], ex.pair(own[1], cur[1]))
        new_store = [dict() for _ in range(P)]
        for x in range(P):
            for k2, v in store[x].items():
                if k2 != cur and k2 != own:
                    new_store[x][k2] = v
            recv = inbox[x][((cur[0] + 1) % P, cur[1])]
            new_store[x][key] = _combine(op, store[x][own], recv) if have_values else None
        store, cur = new_store, key
        run.states.append([[cur]])
        run.combines.append([key])
    run.after_reduction = [cur] if P > 0 else []
    at_place = {cur[0]: cur} if P > 0 else {}
    if have_values and dtype == "bf16" and P > 0:
        for x in range(P):
            store[x][cur] = round_to_bf16(store[x][cur])
    last = cur
    for j in range(P - 1):
        messages, inbox = [], [dict() for _ in range(P)]
        for x in range(P):
            dst = (x + 1) % P
            b = (x - last[0]) % P
            messages.append((x, dst, [(last, block_len[b], itemsize)]))
            inbox[dst][((last[0] + 1) % P, last[1])] = store[x][last]
        run.log.append({"phase": "distribute", "i": j, "N": None, "d": -1, "tx": [last],
                        "messages": messages})
        newkey = ((last[0] + 1) % P, last[1])
        assert newkey[0] not in at_place
        at_place[newkey[0]] = newkey
        for x in range(P):
            store[x][newkey] = inbox[x][newkey]
        last = newkey
    if P > 0:
        assert sorted(at_place) == list(range(P))
    run.out_key = [[at_place[(x - b) % P] for b in range(P)] for x in range(P)]
    if have_values:
        run.outputs = [np.concatenate([store[x][run.out_key[x][b]] for b in range(P)])
                       if P else np.zeros(0) for x in range(P)]
    return run


def allreduce(inputs, steps: int, op: str = "sum", dtype: str = "f32", elements=None,
              group: str = "cyclic"):
    """MPI_Allreduce semantics (Sec. "Introduction"): every process ends with the
    op-reduction of all P input vectors.  Returns the list of P output arrays (over the
    selected elements when ``elements`` is given).

    Pinned by: test_int32_bruteforce, test_float_max_min_exact, test_golden_tree_values.
    """
    P = len(inputs)
    n = len(inputs[0]) if P else 0
    if steps == "ring":
        return simulate_ring(P, n, inputs=inputs, op=op, dtype=dtype, elements=elements).outputs
    return simulate(P, n, steps, inputs=inputs, op=op, dtype=dtype,
                    elements=elements, group=group).outputs


# ---------------------------------------------------------------------------
# Plain definitions used to pin the simulation
# ---------------------------------------------------------------------------

def column_reduce_exact(inputs, op: str, dtype: str):
    """The Allreduce result from its definition, u_{i,Sigma} = u_{i,0} (+) ... (+)
    u_{i,P-1} (Sec. "Combination of distributed data vectors"), for the cases where it
    has a unique value: i32 sum in exact integers reduced mod 2^32 (two's complement),
    and max/min of any type.

    Pinned by: test_column_reduce_exact_brute_force (pure-Python loops).
    """
    stack = np.stack([np.asarray(v) for v in inputs])
    if op == "sum":
        if dtype != "i32":
            raise ValueError("floating-point sums depend on association order")
        tot = stack.astype(np.int64).sum(axis=0)          # exact for P < 2^32
        wrapped = ((tot + 2**31) % 2**32) - 2**31
        return wrapped.astype(np.int32)
    if op == "max":
        return stack.max(axis=0)
    if op == "min":
        return stack.min(axis=0)
    raise ValueError(op)


def kahan_sum_f64(inputs) -> tuple[np.ndarray, np.ndarray]:
    """Compensated (Kahan) sum of the P inputs in rank order, in float64, and the sum
    of absolute values (the scale of the standard summation error bound).

    Pinned by: test_kahan_sum_within_compensated_bound (math.fsum),
    test_kahan_sum_recovers_lost_low_bits, test_planted_kahan_sign_flip_is_caught.
    """
    stack = np.stack([np.asarray(v, dtype=np.float64) for v in inputs])
    s = np.zeros(stack.shape[1], dtype=np.float64)
    comp = np.zeros_like(s)
    for row in stack:
        y = row - comp
        t = s + y
        comp = (t - s) - y
        s = t
    return s, np.abs(stack).sum(axis=0)


# ---------------------------------------------------------------------------
# Cost model (Sec. "Communication model"; eqs. bo_cost, intemediate_cost, lo_cost)
# ---------------------------------------------------------------------------

def cost_model_time(P: int, m_bytes: float, steps, alpha: float, beta: float,
                    gamma: float) -> float:
    """tau for the version with S = steps (eq. bo_cost for r = 0, eq. intemediate_cost
    for 0 < r < L, eq. lo_cost for r = L), with u = m/P.  steps="ring": eq. naive_cost.
    An even S in (2L, 2(P-1)], a fold schedule (reading C19), sends what the
    bandwidth-optimal version sends and combines as often, in S steps.

    Pinned by: test_cost_model_argmin_matches_paper_example,
    test_cost_model_beyond_2L_joins_the_paper_equations,
    test_bandwidth_optimal_traffic.
    """
    L = ceil_log2(P)
    u = m_bytes / P
    if steps == "ring":
        return 2 * (P - 1) * alpha + 2 * (P - 1) * u * beta + (P - 1) * u * gamma
    if 2 * L < steps <= 2 * (P - 1) and steps % 2 == 0:
        return steps * alpha + 2 * (P - 1) * u * beta + (P - 1) * u * gamma
    r = 2 * L - steps
    if not 0 <= r <= L:
        raise ValueError("steps out of range")
    if r == L:
        return L * alpha + P * L * u * beta + P * (2 * L - 2) * u * gamma
    return ((2 * L - r) * alpha
            + (2 * (P - 1) + (2 ** r - 1) * (L - 1)) * u * beta
            + ((P - 1) + (2 ** r - 1) * (2 * L - 2)) * u * gamma)


def optimal_steps(P: int, m_bytes: float, alpha: float, beta: float, gamma: float) -> int:
    """The step count minimising the cost model over integer S in [L, 2L] (eq.
    opt_number_of_steps gives the continuous optimum; reading C15 takes the argmin).

    Pinned by: test_cost_model_argmin_matches_paper_example.
    """
    L = ceil_log2(P)
    if L == 0:
        return 0
    best = None
    for S in range(L, 2 * L + 1):
        t = cost_model_time(P, m_bytes, S, alpha, beta, gamma)
        if best is None or t < best[0] - 1e-18:
            best = (t, S)
    return best[1]
