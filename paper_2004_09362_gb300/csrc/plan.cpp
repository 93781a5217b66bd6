// Host-side schedule builder for the permutation-group Allreduce.
//
// Kolmakov & Zhang, "A Generalization of the Allreduce Operation" (arXiv 2004.09362).
// The builder works in "placement space": a vector at placement p has its block i on
// rank i + p (eq. distr_vector with h = identity and the cyclic group of Table 1a), so
// rank x holds block (x - p) mod P of it, and a move by t^{-d} (eq. bo_dir_perms) keeps
// every block index while the placement drops by d.
//
// Two derived facts about the K shifted copies of the bandwidth-optimal schedule (eq.
// var_starting_set and the equations that follow it) make the builder closed-form:
//  * in copy s at step i, the vector with index k >= 1 sits at placement s + k and
//    its content depends only on that placement; the index-0 vector (q*, eq.
//    bo_starting_set) has its own content.  So the union of all copies holds exactly
//    one q' per placement in [1, K + N_i - 2] and one q* per placement in [0, K); q*_s
//    equals q'_s (same content, same association tree) until the first step with odd
//    N_i, after which the two are different vectors (Sec. "Latency-optimal version":
//    q* and q' cannot be combined even if they have the same placement).
//  * step i transmits the q' at placements [ceil(N_i/2), K + N_i - 2] (taken mod P),
//    i.e. min(P, K - 1 + floor(N_i/2)) blocks per rank (eq. bo_tx_dist, plus the one
//    extra vector t^{N_i} q'_{N_i} per added copy, Sec. "Moving towards latency-optimal
//    version"), and each received vector is combined into the q' and/or q* at its new
//    placement.
// With the self-inverse group of Table 1b (P a power of two) every "+" on placements and
// ranks becomes XOR: placement p puts block i on rank i ^ p, the step operator is
// t_{N_i/2} (x -> x ^ N_i/2), copy s has index k at placement s ^ k, and the unions of
// the copies' placement sets are enumerated instead of taken as ranges.
// Beyond 2L steps (cyclic group): fold schedules generalize the bandwidth-optimal step
// from folding floor(N_i/2) vectors to folding f_i of them by t^{-f_i} (build_folds),
// and the Ring moves one vector per step by the generator t (build_ring).
#include <algorithm>
#include <map>
#include <stdexcept>
#include <utility>

#include "gar_internal.hpp"

namespace gar {

int elem_size(int dtype) { return dtype == GAR_BF16 ? 2 : 4; }
int acc_size(int) { return 4; }

int ceil_log2(int P) {
  int L = 0;
  while ((1 << L) < P) ++L;
  return L;
}

namespace {

// Placements lo, lo+1, ..., hi taken mod P, each once, in first-appearance order.
std::vector<int32_t> placement_range(long lo, long hi, int P) {
  std::vector<int32_t> out;
  if (hi < lo) return out;
  std::vector<char> seen(P, 0);
  for (long t = lo; t <= hi && (long)out.size() < P; ++t) {
    const int p = (int)(((t % P) + P) % P);
    if (!seen[p]) {
      seen[p] = 1;
      out.push_back(p);
    }
  }
  return out;
}

// Group operation t_a(b) and inverse on {0..P-1}: cyclic (Table 1a) or XOR (Table 1b).
struct Group {
  int P;
  bool xr;
  int op(int a, int b) const { return xr ? (a ^ b) : (a + b) % P; }
  int inv(int a) const { return xr ? a : (P - a) % P; }
};

// Placements t_s(k) for s in [0, K), k in [lo, hi], each once.  Cyclic: the
// consecutive range [lo, K - 1 + hi] mod P (placement_range); XOR: enumerated.
std::vector<int32_t> union_placements(const Group &g, int K, long lo, long hi) {
  if (!g.xr) return placement_range(lo, (long)K - 1 + hi, g.P);
  std::vector<int32_t> out;
  if (hi < lo) return out;
  std::vector<char> seen(g.P, 0);
  for (int s = 0; s < K; ++s)
    for (long k = lo; k <= hi; ++k) {
      const int p = g.op(s, (int)k);
      if (!seen[p]) {
        seen[p] = 1;
        out.push_back(p);
      }
    }
  return out;
}

StepOp make_op(int recv_place, int dst_place, Buf recv_buf) {
  StepOp op{};
  op.recv_place = (int16_t)recv_place;
  op.dst_place = (int16_t)dst_place;
  op.recv_buf = recv_buf;
  op.out0_buf = op.out0_own = op.out1_buf = op.out1_own = BUF_NONE;
  return op;
}

void add_out(StepOp &op, Buf dst, Buf own) {
  if (op.out0_buf == BUF_NONE) {
    op.out0_buf = dst;
    op.out0_own = own;
  } else if (op.out1_buf == BUF_NONE) {
    op.out1_buf = dst;
    op.out1_own = own;
  } else {
    throw std::logic_error("block op with more than two outputs");
  }
}

// Step-faithful schedule: one launch per communication step.  Storage per rank:
//  - K == 1 (bandwidth-optimal): the transmit placements [ceil(N/2), N-1] and the
//    combine placements [N mod 2, ceil(N/2)-1] are disjoint, so every step runs in
//    place -- in the rank buffer itself when the accumulation type is the element
//    type, else in one fp32 workspace slice filled by step 0.  q*_0 (placement 0,
//    block x) is never a q' slot.
//  - K > 1: transmit and combine placements overlap, so q' slots ping-pong between two
//    workspace slices (the partner reads the old slice while the new one is written);
//    q* slots live in a third slice once they stop aliasing q'.
// Results are written to the rank buffers by the last reduction step; the distribution
// steps copy partner blocks rank buffer to rank buffer (senders [N mod 2, ceil(N/2)-1]
// and receivers [ceil(N/2), N-1] are disjoint placements).
void build_step_faithful(gar_plan *pl) {
  const int P = pl->P, L = pl->L, K = pl->K, r = pl->r;
  const Group g{P, pl->group == GAR_GROUP_XOR};
  const bool acc_is_elem = pl->dtype != GAR_BF16;
  const Buf inplace = acc_is_elem ? BUF_RANK : BUF_QP0;
  const Buf qs_loc = (K == 1) ? inplace : BUF_QS;
  bool aliased = true;
  Buf finalize_from = BUF_NONE;

  for (int i = 0; i < L; ++i) {
    const int N = pl->N[i], d = N / 2, c = N - d;
    const bool last = (i == L - 1), even = (N % 2 == 0);
    const Buf src = (i == 0) ? BUF_RANK
                             : (K == 1 ? inplace : (((i - 1) % 2 == 0) ? BUF_QP0 : BUF_QP1));
    const Buf dst = (K == 1) ? inplace : ((i % 2 == 0) ? BUF_QP0 : BUF_QP1);
    // Results go straight to the rank buffers, except when this step still reads them
    // as transmit sources and K > 1 (only P == 2, K == 2): then stage and copy after.
    Buf fin = BUF_RANK;
    if (last && K > 1 && src == BUF_RANK) {
      fin = dst;
      finalize_from = dst;
    }
    std::vector<char> in_next(P, 0);  // q' placements alive after this step
    if (c >= 2)
      for (int32_t p : union_placements(g, K, 1, c - 1)) in_next[p] = 1;

    CommStep cs;
    cs.phase = 0;
    cs.i = i;
    cs.N = N;
    cs.d = d;
    cs.partner = d;  // receive from the rank the step operator t_d^{-1} maps onto x
    cs.tx = union_placements(g, K, c, N - 1);
    Launch ln;
    ln.phase = 0;
    ln.comm_step = (int)pl->comm.size();
    ln.partner = d;
    ln.first_op = (int)pl->ops.size();
    for (int32_t p : cs.tx) {
      const int pp = g.op(p, g.inv(d));  // placement after the move by t_d^{-1}
      const bool to_qp = in_next[pp] != 0;
      const bool to_qs = even && pp < K;
      StepOp op = make_op(p, pp, src);
      if (aliased) {
        // q*_pp and q'_pp are one vector: one combine serves both
        if (even && to_qs)
          add_out(op, last ? fin : dst, src);
        else if (to_qp)
          add_out(op, dst, src);
      } else {
        if (to_qp) add_out(op, dst, src);
        if (to_qs) add_out(op, last ? fin : qs_loc, qs_loc);
      }
      if (op.out0_buf == BUF_NONE) throw std::logic_error("transmitted vector has no use");
      pl->ops.push_back(op);
    }
    if (aliased && !even) {
      // First odd N_i: q*_s sits this step out (eq. bo_step_odd) while q'_s is combined,
      // so q*_s gets storage of its own now.
      if (!(K == 1 && src == qs_loc)) {
        for (int s = 0; s < K; ++s) {
          StepOp op = make_op(-1, s, BUF_NONE);
          add_out(op, qs_loc, src);
          pl->ops.push_back(op);
        }
      }
      aliased = false;
    }
    ln.nops = (int)pl->ops.size() - ln.first_op;
    cs.msg_bytes = (uint64_t)cs.tx.size() * pl->n *
                   (uint64_t)(src == BUF_RANK ? elem_size(pl->dtype) : acc_size(pl->dtype));
    pl->comm.push_back(cs);
    pl->launches.push_back(ln);
  }

  if (finalize_from != BUF_NONE) {
    Launch ln;
    ln.phase = 2;
    ln.comm_step = -1;
    ln.partner = 0;
    ln.first_op = (int)pl->ops.size();
    for (int s = 0; s < K; ++s) {
      StepOp op = make_op(-1, s, BUF_NONE);
      add_out(op, BUF_RANK, finalize_from);
      pl->ops.push_back(op);
    }
    ln.nops = K;
    pl->launches.push_back(ln);
  }

  // Distribution phase: reduction steps L-r-1 .. 0 reversed, no combination.
  for (int i = L - r - 1; i >= 0; --i) {
    const int N = pl->N[i], d = N / 2, c = N - d;
    CommStep cs;
    cs.phase = 1;
    cs.i = i;
    cs.N = N;
    cs.d = d;
    cs.partner = g.xr ? d : -d;  // receive from t_d^{-1}(x): x - d, or x XOR d
    Launch ln;
    ln.phase = 1;
    ln.comm_step = (int)pl->comm.size();
    ln.partner = cs.partner;
    ln.first_op = (int)pl->ops.size();
    for (int p = N % 2; p < c; ++p) {
      cs.tx.push_back(p);
      StepOp op = make_op(p, g.op(p, d), BUF_RANK);
      add_out(op, BUF_RANK, BUF_NONE);
      pl->ops.push_back(op);
    }
    ln.nops = (int)pl->ops.size() - ln.first_op;
    cs.msg_bytes = (uint64_t)cs.tx.size() * pl->n * (uint64_t)elem_size(pl->dtype);
    pl->comm.push_back(cs);
    pl->launches.push_back(ln);
  }

  for (const StepOp &op : pl->ops) {
    for (uint8_t b : {op.recv_buf, op.out0_buf, op.out0_own, op.out1_buf, op.out1_own})
      if (b >= BUF_QP0) pl->ws_used[b - BUF_QP0] = true;
  }
}

// Fused program: the same placement-space schedule evaluated for one element position
// whose P contributions are rotated by its block b (value j = rank (b + j) mod P).  Each
// combine "own (+) received" becomes one SSA value; identical (own, received) pairs are
// one value (the union of the shifted copies computes every distinct vector once).
void build_fused(gar_plan *pl) {
  const int P = pl->P, L = pl->L, K = pl->K, r = pl->r;
  const Group g{P, pl->group == GAR_GROUP_XOR};
  FusedProgram &fp = pl->prog;
  fp = FusedProgram{};
  fp.P = P;
  fp.K = K;
  std::map<std::pair<int, int>, int> cse;
  std::vector<int32_t> A, B, PL;
  std::vector<int8_t> ST;
  auto mk = [&](int a, int b, int place, int star) {
    if (a < 0 || b < 0) throw std::logic_error("fused program reads a dead vector");
    auto key = std::make_pair(a, b);
    auto it = cse.find(key);
    if (it != cse.end()) {
      if (PL[it->second - P] != place) throw std::logic_error("one vector at two placements");
      return it->second;
    }
    const int id = P + (int)A.size();
    A.push_back(a);
    B.push_back(b);
    PL.push_back(place);
    ST.push_back((int8_t)star);
    cse.emplace(key, id);
    return id;
  };
  std::vector<int> qp(P), qs(K);
  for (int p = 0; p < P; ++p) qp[p] = p;
  for (int s = 0; s < K; ++s) qs[s] = s;
  for (int i = 0; i < L; ++i) {
    const int N = pl->N[i], d = N / 2, c = N - d;
    const bool even = (N % 2 == 0);
    std::vector<int> nqp(P, -1), nqs(K);
    // q*_s first, then q'_p: the values are CSE'd, the order only fixes numbering
    // the vector received at placement p came from placement t_d(p)
    for (int s = 0; s < K; ++s) nqs[s] = even ? mk(qs[s], qp[g.op(s, d)], s, 1) : qs[s];
    if (c >= 2)
      for (int32_t p : union_placements(g, K, 1, c - 1)) nqp[p] = mk(qp[p], qp[g.op(p, d)], p, 0);
    qp.swap(nqp);
    qs.swap(nqs);
  }
  // Keep only the combines the K results need.
  const int nall = (int)A.size();
  std::vector<char> live(P + nall, 0);
  std::vector<int> stack(qs.begin(), qs.end());
  while (!stack.empty()) {
    const int v = stack.back();
    stack.pop_back();
    if (live[v]) continue;
    live[v] = 1;
    if (v >= P) {
      stack.push_back(A[v - P]);
      stack.push_back(B[v - P]);
    }
  }
  std::vector<int> renum(P + nall, -1);
  for (int v = 0; v < P; ++v) renum[v] = v;
  for (int k = 0; k < nall; ++k) {
    if (!live[P + k]) continue;
    renum[P + k] = P + (int)fp.a.size();
    fp.a.push_back(renum[A[k]]);
    fp.b.push_back(renum[B[k]]);
    fp.place.push_back(PL[k]);
    fp.star.push_back(ST[k]);
  }
  for (int s = 0; s < K; ++s) fp.out.push_back(renum[qs[s]]);
  // Origins: copy s sits at placement s; distribution step i (reversed) copies
  // placements [N mod 2, ceil(N/2)-1] to +floor(N/2).
  fp.origin.assign(P, -1);
  for (int s = 0; s < K; ++s) fp.origin[s] = s;
  for (int i = L - r - 1; i >= 0; --i) {
    const int N = pl->N[i], d = N / 2, c = N - d;
    for (int p = N % 2; p < c; ++p) fp.origin[g.op(p, d)] = fp.origin[p];
  }
  for (int p = 0; p < P; ++p)
    if (fp.origin[p] < 0) throw std::logic_error("placement without a result");
}

// Fold counts for F reduction steps (F > L): a step with N vectors folds f of them, the
// ones with index [N-f, N), by t^{-f} onto [N-2f, N-f); f = floor(N/2) is the
// bandwidth-optimal step.  The P-1 folds are spread as evenly as 1 <= f <= floor(N/2)
// and reachability (the remaining steps, halving, must still get to N = 1) allow.
std::vector<int> fold_counts(int P, int F) {
  std::vector<int> folds;
  int N = P;
  for (int i = 0; i < F; ++i) {
    const int r = F - i;
    const long long pow2 = (r - 1 >= 31) ? (1LL << 31) : (1LL << (r - 1));
    const int lo = (int)std::max<long long>(1, (long long)N - pow2);
    const int hi = std::min(N / 2, N - r);
    const int want = (N - 1 + r - 1) / r;  // ceil((N - 1) / r)
    const int f = std::min(std::max(want, lo), hi);
    folds.push_back(f);
    N -= f;
  }
  if (N != 1) throw std::logic_error("fold schedule does not end with one vector");
  return folds;
}

// Fold schedule (S = 2F > 2L, one result copy): step-faithful ops run in place like the
// bandwidth-optimal schedule (transmitted [N-f, N) and combined [N-2f, N-f) placements
// never overlap); placements [0, N-2f) sit the step out.  With a wider accumulation type
// (bf16 -> fp32) a placement keeps its input in the rank buffer, and is sent in the
// element type, until it is first combined; the combination lands in the fp32 slice.
void build_folds(gar_plan *pl) {
  const int P = pl->P;
  const int F = (int)pl->folds.size();
  const Buf inplace = pl->dtype != GAR_BF16 ? BUF_RANK : BUF_QP0;
  std::vector<int> Ns{P};
  for (int f : pl->folds) Ns.push_back(Ns.back() - f);
  std::vector<Buf> loc(P, BUF_RANK);  // where each placement's vector lives now
  for (int i = 0; i < F; ++i) {
    const int N = Ns[i], f = pl->folds[i];
    const bool last = (i == F - 1);
    CommStep cs;
    cs.phase = 0;
    cs.i = i;
    cs.N = N;
    cs.d = f;
    cs.partner = f;
    cs.msg_bytes = 0;
    Launch ln;
    ln.phase = 0;
    ln.comm_step = (int)pl->comm.size();
    ln.partner = f;
    ln.first_op = (int)pl->ops.size();
    for (int p = N - f; p < N; ++p) {
      cs.tx.push_back(p);
      StepOp op = make_op(p, p - f, loc[p]);
      add_out(op, last ? BUF_RANK : inplace, loc[p - f]);
      pl->ops.push_back(op);
      cs.msg_bytes += (uint64_t)pl->n *
                      (uint64_t)(loc[p] == BUF_RANK ? elem_size(pl->dtype) : acc_size(pl->dtype));
    }
    for (int p = N - 2 * f; p < N - f; ++p) loc[p] = inplace;
    ln.nops = (int)pl->ops.size() - ln.first_op;
    pl->comm.push_back(cs);
    pl->launches.push_back(ln);
  }
  for (int i = F - 1; i >= 0; --i) {
    const int N = Ns[i], f = pl->folds[i];
    CommStep cs;
    cs.phase = 1;
    cs.i = i;
    cs.N = N;
    cs.d = f;
    cs.partner = -f;
    Launch ln;
    ln.phase = 1;
    ln.comm_step = (int)pl->comm.size();
    ln.partner = -f;
    ln.first_op = (int)pl->ops.size();
    for (int p = N - 2 * f; p < N - f; ++p) {
      cs.tx.push_back(p);
      StepOp op = make_op(p, p + f, BUF_RANK);
      add_out(op, BUF_RANK, BUF_NONE);
      pl->ops.push_back(op);
    }
    ln.nops = (int)pl->ops.size() - ln.first_op;
    cs.msg_bytes = (uint64_t)f * pl->n * (uint64_t)elem_size(pl->dtype);
    pl->comm.push_back(cs);
    pl->launches.push_back(ln);
  }
  for (const StepOp &op : pl->ops)
    for (uint8_t b : {op.recv_buf, op.out0_buf, op.out0_own, op.out1_buf, op.out1_own})
      if (b >= BUF_QP0) pl->ws_used[b - BUF_QP0] = true;
  FusedProgram &fp = pl->prog;
  fp = FusedProgram{};
  fp.P = P;
  fp.K = 1;
  std::vector<int> qp(P);
  for (int p = 0; p < P; ++p) qp[p] = p;
  for (int i = 0; i < F; ++i) {
    const int N = Ns[i], f = pl->folds[i];
    for (int k = N - 2 * f; k < N - f; ++k) {
      fp.a.push_back(qp[k]);
      fp.b.push_back(qp[k + f]);
      fp.place.push_back(k);
      fp.star.push_back(0);
      qp[k] = P + (int)fp.a.size() - 1;
    }
  }
  fp.out.push_back(qp[0]);
  fp.origin.assign(P, 0);
}

// The Ring (Sec. "Allreduce as permutation composition", cyclic group: the operator of
// every step is the generator t, x -> x + 1).  Reduction step i moves the partial at
// placement i to placement i + 1 and combines it there with the rank's own initial block
// (eq. ring_reduce); distribution step j moves the copy at placement P-1+j on by one.
// In place: step i writes placement i + 1 while the partner reads placement i.
void build_ring(gar_plan *pl) {
  const int P = pl->P;
  const bool acc_is_elem = pl->dtype != GAR_BF16;
  const Buf partial = acc_is_elem ? BUF_RANK : BUF_QP0;
  for (int i = 0; i + 1 < P; ++i) {
    const bool last = (i + 2 == P);
    const Buf src = (i == 0) ? BUF_RANK : partial;
    CommStep cs;
    cs.phase = 0;
    cs.i = i;
    cs.N = 0;
    cs.d = 1;
    cs.partner = -1;
    cs.tx = {i};
    Launch ln;
    ln.phase = 0;
    ln.comm_step = (int)pl->comm.size();
    ln.partner = -1;
    ln.first_op = (int)pl->ops.size();
    StepOp op = make_op(i, i + 1, src);
    add_out(op, last ? BUF_RANK : partial, BUF_RANK);   // own initial block (+) received partial
    pl->ops.push_back(op);
    ln.nops = 1;
    cs.msg_bytes = pl->n * (uint64_t)(src == BUF_RANK ? elem_size(pl->dtype) : acc_size(pl->dtype));
    pl->comm.push_back(cs);
    pl->launches.push_back(ln);
  }
  for (int j = 0; j + 1 < P; ++j) {
    const int from = (P - 1 + j) % P, to = j;
    CommStep cs;
    cs.phase = 1;
    cs.i = j;
    cs.N = 0;
    cs.d = 1;
    cs.partner = -1;
    cs.tx = {from};
    Launch ln;
    ln.phase = 1;
    ln.comm_step = (int)pl->comm.size();
    ln.partner = -1;
    ln.first_op = (int)pl->ops.size();
    StepOp op = make_op(from, to, BUF_RANK);
    add_out(op, BUF_RANK, BUF_NONE);
    pl->ops.push_back(op);
    ln.nops = 1;
    cs.msg_bytes = pl->n * (uint64_t)elem_size(pl->dtype);
    pl->comm.push_back(cs);
    pl->launches.push_back(ln);
  }
  for (const StepOp &op : pl->ops)
    for (uint8_t b : {op.recv_buf, op.out0_buf, op.out0_own, op.out1_buf, op.out1_own})
      if (b >= BUF_QP0) pl->ws_used[b - BUF_QP0] = true;
  // fused program: the chain q_{P-1} (+) (... (+) (q_1 (+) q_0)), written to every rank
  FusedProgram &fp = pl->prog;
  fp = FusedProgram{};
  fp.P = P;
  fp.K = 1;
  int v = 0;
  for (int k = 1; k < P; ++k) {
    fp.a.push_back(k);
    fp.b.push_back(v);
    fp.place.push_back(k);
    fp.star.push_back(0);
    v = P + (int)fp.a.size() - 1;
  }
  fp.out.push_back(v);
  fp.origin.assign(P, 0);
}

}  // namespace

int build_plan(gar_plan *pl) {
  const int P = pl->P;
  pl->L = ceil_log2(P);
  pl->N.clear();
  pl->N.push_back(P);
  while (pl->N.back() > 1) pl->N.push_back((pl->N.back() + 1) / 2);
  if ((int)pl->N.size() != pl->L + 1) return GAR_EINVAL;
  if (pl->ring) {
    pl->r = 0;
    pl->K = 1;
  } else if (pl->S > 2 * pl->L) {
    pl->r = 0;
    pl->K = 1;
    try {
      pl->folds = fold_counts(P, pl->S / 2);
    } catch (const std::exception &e) {
      set_error(std::string("schedule builder: ") + e.what());
      return GAR_EINVAL;
    }
  } else {
    pl->r = 2 * pl->L - pl->S;
    if (pl->r < 0 || pl->r > pl->L) return GAR_EINVAL;
    pl->K = pl->N[pl->L - pl->r];
  }
  pl->q = pl->n / (uint64_t)P;
  pl->rem = pl->n % (uint64_t)P;
  pl->comm.clear();
  pl->ops.clear();
  pl->launches.clear();
  try {
    if (pl->ring) {
      build_ring(pl);
    } else if (!pl->folds.empty()) {
      build_folds(pl);
    } else {
      build_step_faithful(pl);
      build_fused(pl);
    }
  } catch (const std::exception &e) {
    set_error(std::string("schedule builder: ") + e.what());
    return GAR_EINVAL;
  }
  if ((int)pl->comm.size() != pl->S) {
    set_error("schedule builder: step count mismatch");
    return GAR_EINVAL;
  }
  pl->n_pad = (pl->n + 63) / 64 * 64;
  int nslices = 0;
  for (bool u : pl->ws_used) nslices += u ? 1 : 0;
  pl->ws_bytes = (size_t)nslices * (size_t)P * (size_t)pl->n_pad * (size_t)acc_size(pl->dtype);
  return GAR_OK;
}

}  // namespace gar
