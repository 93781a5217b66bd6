/*
 * gar.h -- permutation-group Allreduce on one GB300 (sm_103a).
 *
 * Implements the generalized Allreduce of D. Kolmakov and X. Zhang, "A Generalization
 * of the Allreduce Operation" (arXiv 2004.09362): the schedule built from a
 * permutation group T_P (the cyclic group for any P, including non-powers of two and
 * primes; the XOR group of Table 1b for powers of two), with a step count S that can be
 * set anywhere from ceil(log2 P) (latency-optimal, Sec. "Latency-optimal version") to
 * 2 ceil(log2 P) (bandwidth-optimal, Sec. "Bandwidth-optimal algorithm"; between them
 * Sec. "Moving towards latency-optimal version"), and beyond that up to the Ring's
 * 2(P-1) steps (fold schedules, GAR_STEPS_RING).
 *
 * The P processes of the paper are P "virtual ranks": P equally sized vectors that
 * all live in the memory of one GPU.  A message of the paper is a read of the partner
 * rank's block.  Semantics follow MPI_Allreduce with MPI_IN_PLACE (Sec.
 * "Introduction"): after the call every rank buffer holds the op-reduction of all P
 * input vectors.
 *
 * Conventions for every function below:
 *  - Return value: GAR_OK (0) on success, a negative GAR_E* code otherwise.  No error
 *    is raised asynchronously by the library itself; a CUDA error from an earlier
 *    kernel surfaces as GAR_ECUDA from the next call that checks.  gar_strerror()
 *    names a code; gar_last_error() gives the calling thread's last detail message.
 *  - Ownership: rank buffers, workspaces and batch descriptor arrays belong to the
 *    caller.  A plan owns its host tables and the small device tables it uploads
 *    (descriptors, byte counters); gar_plan_destroy frees them.
 *  - Ordering: functions taking a stream enqueue work on it and return without
 *    waiting, except where stated.  A plan may be used from one host thread at a time.
 *  - Device pointers must point into memory of the current CUDA device.
 */
#ifndef GAR_H
#define GAR_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define GAR_API __attribute__((visibility("default")))
#else
#define GAR_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct gar_plan gar_plan;
typedef struct CUstream_st *gar_stream_t; /* identical to cudaStream_t */

/* Element types.  GAR_BF16 combines in fp32 and rounds once to bf16 (round to
 * nearest even) when a result is written. */
enum { GAR_F32 = 0, GAR_BF16 = 1, GAR_I32 = 2 };

/* Reduction operators.  Only commutative operators: the method reorders operands
 * (Sec. "Related work" names commutativity as the condition for cyclic patterns).
 * GAR_SUM on GAR_I32 wraps modulo 2^32. */
enum { GAR_SUM = 0, GAR_MAX = 1, GAR_MIN = 2 };

/* Execution modes.
 * GAR_STEP_FAITHFUL: one kernel launch per schedule step; a step reads the
 *   partner rank's blocks (the paper's send/receive) with 16-byte vector loads and
 *   combines them with the own block; needs the workspace reported by
 *   gar_plan_bytes; records the bytes read from partners per step.  The launches of
 *   one call are chained by programmatic dependent launch: a launch may become resident
 *   early but reads nothing before every earlier kernel on the stream has completed.
 * GAR_FUSED: one launch for the whole Allreduce; per element position the P
 *   contributions are loaded once, the reduction program that the schedule induces
 *   runs in registers, and every rank's result is written once.  The program becomes
 *   straight-line code compiled at run time, so fused mode takes programs of at most
 *   GAR_FUSED_MAX_OPS operations (combines + P loads + P stores; the compile of the
 *   largest takes about a minute on one core, and it grows faster than linearly).
 *   Larger programs -- latency-optimal schedules at a few hundred ranks and up -- make
 *   every fused call return GAR_EINVAL; GAR_STEP_FAITHFUL runs any plan.
 * GAR_STEP_PERSISTENT: the step-faithful schedule in one cooperative launch; a
 *   grid-wide barrier separates the steps instead of a kernel boundary.  Every barrier
 *   wait is bounded (gar_plan_debug_barrier): a CTA that waits too long records a
 *   timeout and returns, every other CTA stops at its next poll, and
 *   gar_plan_status reports GAR_ETIMEOUT.  Same workspace and results as
 *   GAR_STEP_FAITHFUL. */
enum { GAR_STEP_FAITHFUL = 0, GAR_FUSED = 1, GAR_STEP_PERSISTENT = 2 };
#define GAR_FUSED_MAX_OPS 4096

/* The permutation group T_P (Sec. "Communication description via permutations").
 * GAR_GROUP_CYCLIC: t_k(x) = x + k mod P (Table 1a), any P.
 * GAR_GROUP_XOR: t_k(x) = x XOR k, the self-inverse group of Table 1b, P a power of two;
 *   the bandwidth-optimal schedule is then Recursive Halving and the latency-optimal one
 *   Recursive Doubling (every step a pairwise exchange with rank x XOR N_i/2). */
enum { GAR_GROUP_CYCLIC = 0, GAR_GROUP_XOR = 1 };

/* Special values for the `steps` argument of gar_plan_create. */
#define GAR_STEPS_BO (-1) /* 2 ceil(log2 P): bandwidth-optimal */
#define GAR_STEPS_LO (-2) /* ceil(log2 P): latency-optimal */
/* The Ring: the straightforward algorithm of Sec. "Allreduce as permutation composition"
 * with the cyclic group, every step moving by the generator t (x -> x + 1); 2(P-1) steps
 * (eq. naive_cost), the far end of the paper's step range.  Cyclic group only. */
#define GAR_STEPS_RING (-3)

#define GAR_MAX_P 1024 /* largest supported number of virtual ranks */

enum {
  GAR_OK = 0,
  GAR_EINVAL = -1,  /* bad argument (P, n, dtype, op, steps, mode, null pointer) */
  GAR_ENOMEM = -2,  /* host or device allocation failed */
  GAR_EALIGN = -3,  /* a buffer is not 16-byte aligned */
  GAR_ECUDA = -4,   /* a CUDA runtime call failed (detail in gar_last_error) */
  GAR_EJIT = -5,    /* run-time compilation of a specialized kernel failed */
  GAR_ENOWS = -6,   /* step-faithful mode needs a workspace that was not set or is too small */
  GAR_ESTATE = -7,  /* operation not valid in the plan's current state */
  GAR_ETIMEOUT = -8 /* a bounded wait inside a kernel gave up (gar_plan_status) */
};

/* Describes a plan.  Symbols follow the paper: L = ceil(log2 P) reduction steps
 * (eq. bo_starting_set_size), S = 2L - r total steps, K = number of q_Sigma copies at
 * the end of the reduction phase (K = N_{L-r}; K = 1 bandwidth-optimal, K = P
 * latency-optimal).  Fold schedules and the Ring have S > 2L, r = 0 and K = 1. */
typedef struct {
  int32_t P;
  int32_t L;
  int32_t S;
  int32_t r;
  int32_t K;
  int32_t dtype;
  int32_t op;
  int32_t n_launches;        /* step-faithful kernel launches per Allreduce */
  uint64_t n;                /* elements per rank */
  int32_t fused_combines;    /* combines per element position in fused mode */
  int32_t fused_width;       /* elements per thread-vector in the fused kernel (0 until compiled) */
  int32_t fused_regs;        /* registers per thread of the loaded fused kernel (0 until loaded) */
  int32_t fused_local_bytes; /* local (spill) bytes per thread of the loaded fused kernel */
  int32_t group;             /* GAR_GROUP_CYCLIC or GAR_GROUP_XOR */
  int32_t ring;              /* 1 for the Ring schedule (GAR_STEPS_RING) */
  int32_t fused_form;        /* fused kernel the plan uses: GAR_FORM_SINGLE, _BREADTH or _SPLIT */
} gar_plan_info;

/* Values of gar_plan_info.fused_form.  GAR_FORM_SINGLE: each thread evaluates the whole
 * program result by result for 1..8 element positions.  GAR_FORM_BREADTH: each thread
 * evaluates it step by step for one element position, with paired fp32 adds (the widest
 * programs in two passes over halves of the result copies, recomputing the values both
 * halves need); taken by float sums with several result copies whose single-thread form
 * would keep more than 160 values alive per element position (large latency-optimal and
 * near-latency-optimal schedules, e.g. P = 127 at S = 7 and 8).  GAR_FORM_SPLIT: two lanes of a warp share
 * an element position, each evaluating the combines of half the placements and
 * receiving the vectors a step moves across the halves by a warp shuffle; defined for
 * latency-optimal cyclic schedules (every placement holds its own result copy) and
 * taken only when forced (environment GAR_TUNE_FUSED_FORM=2): on GB300 it was slower
 * than the breadth-first form.  All forms give the same bits. */
enum { GAR_FORM_SINGLE = 0, GAR_FORM_BREADTH = 1, GAR_FORM_SPLIT = 2 };

/* Creates a schedule for P virtual ranks of n elements each.
 * P: 1..GAR_MAX_P.  n: elements per rank (0 is allowed: every call is a no-op).
 * steps: S in [ceil(log2 P), 2 ceil(log2 P)], or GAR_STEPS_BO / GAR_STEPS_LO /
 * GAR_STEPS_RING, or an even S in (2 ceil(log2 P), 2(P-1)] (cyclic group): a fold
 * schedule, which generalizes the bandwidth-optimal step from folding floor(N_i/2)
 * vectors to folding f_i <= floor(N_i/2) of them by t^{-f_i}, with the P-1 folds spread
 * evenly over S/2 steps -- every such S moves the bandwidth-optimal 2(P-1) blocks per
 * rank in smaller pieces (the step counts Sec. "Conclusion" leaves to future work).
 * The block partition is the paper's V_j = (u_{0,j}, ..., u_{P-1,j}) (eq.
 * initial_data) with the first n mod P blocks one element longer.  Host-only: needs
 * no GPU.  *out is set only on success. */
GAR_API int gar_plan_create(gar_plan **out, int P, uint64_t n, int dtype, int op, int steps);

/* gar_plan_create with an explicit group T_P (GAR_GROUP_*); gar_plan_create uses the
 * cyclic group.  GAR_GROUP_XOR with P not a power of two returns GAR_EINVAL.  With the
 * XOR group, K = 2^r result copies (r = 2L - S): the intermediate step counts are the
 * Recursive Halving / Recursive Doubling hybrid. */
GAR_API int gar_plan_create_group(gar_plan **out, int P, uint64_t n, int dtype, int op, int steps,
                                  int group);

/* Frees the plan and its device tables.  NULL is a no-op.  The caller must make sure
 * no work using the plan is still running.  (Resource management; no counterpart in the
 * paper.) */
GAR_API void gar_plan_destroy(gar_plan *plan);

/* Fills *info (see gar_plan_info).  Host-only. */
GAR_API int gar_plan_get_info(const gar_plan *plan, gar_plan_info *info);

/* Sizes.  workspace_bytes: device workspace step-faithful mode needs (0 when the
 * schedule runs in place: bandwidth-optimal, fold and Ring schedules in f32/i32).  msg_bytes_per_step (may be
 * NULL, else S entries): bytes all ranks together read from their partners in each
 * communication step, the schedule's message volume (Sec. "Communication
 * operator": every rank sends its blocks of the transmitted vectors).  S (may be
 * NULL) receives the step count.  Host-only. */
GAR_API int gar_plan_bytes(const gar_plan *plan, size_t *workspace_bytes,
                   uint64_t *msg_bytes_per_step, int *S);

/* Schedule introspection (host-only).  For communication step t in [0, S):
 * phase = 0 (reduction) or 1 (distribution); partner: rank x receives from rank
 * (x + partner) mod P in the cyclic group (reduction: +floor(N_i/2), eq. bo_dir_perms;
 * distribution: -floor(N_i/2); fold schedules: +f_i and -f_i, f_i the vectors folded
 * in reduction step i; the Ring: -1 in both phases) and from rank x XOR
 * partner in the XOR group; placements[0..*count) = placements of the vectors each rank
 * transmits (eq. bo_tx_dist and its shifted forms).  placements may be NULL to query
 * the count; otherwise it must hold P entries. */
GAR_API int gar_plan_step(const gar_plan *plan, int t, int *phase, int *partner,
                  int32_t *placements, int *count);

/* origin[p] for p in [0, P): the result copy (0..K-1) that placement p receives in the
 * distribution phase (end of Sec. "Bandwidth-optimal algorithm").  Rank x's result for
 * block b is at placement (x - b) mod P (cyclic group) or x XOR b (XOR group). */
GAR_API int gar_plan_origin(const gar_plan *plan, int32_t *origin);

/* The fused-mode program: value ids 0..P-1 are the P contributions of an element
 * position in block b, contribution j coming from rank t_j(b) ((b + j) mod P, or b XOR j
 * in the XOR group); combine k makes value P + k = ops[2k] (+) ops[2k+1] (own,
 * received; eq. distr_vectors_combination).  outputs[s] (s < K) = value id of result
 * copy s.  Pass NULL arrays to query *nops; ops must hold 2 * *nops entries and outputs
 * K entries. */
GAR_API int gar_plan_fused_program(const gar_plan *plan, int32_t *ops, int *nops, int32_t *outputs);

/* The step-faithful op table (host-only, for inspection and tests).  Each op is 8
 * int32: {launch, recv_place, dst_place, recv_buf, out0_buf, out0_own, out1_buf,
 * out1_own}; buffers: 0 none, 1 rank buffer, 2 q' ping, 3 q' pong, 4 q* store.
 * launch_partner[l] = receive offset of launch l.  Query *nops with ops == NULL. */
GAR_API int gar_plan_step_ops(const gar_plan *plan, int32_t *ops, int *nops, int32_t *launch_partner,
                      int *nlaunch);

/* Caller-owned device workspace for step-faithful mode (16-byte aligned, at least
 * workspace_bytes): the storage of the partial vectors q' and q* that the paper's
 * processes keep between steps (Sec. "Latency-optimal version" keeps the two apart).
 * The memory model has no counterpart in the paper.  NULL with 0 bytes detaches it.
 * GAR_EALIGN for a misaligned pointer. */
GAR_API int gar_plan_set_workspace(gar_plan *plan, void *dev_ptr, size_t bytes);

/* The CUDA C source of the plan's generated fused kernel (host-only): of the kernel the
 * plan runs once it is prepared (gar_plan_prepare or a first fused call, which rebuild a
 * kernel of more than 128 registers in 64-thread CTAs), else of its first compile.
 * Copies at most
 * *len bytes (including the terminating NUL) to buf and sets *len to the full size
 * including the NUL; pass buf == NULL to query the size. */
GAR_API int gar_plan_fused_source(const gar_plan *plan, char *buf, size_t *len);

/* Compiles (host-only, needs no GPU) the specialized kernel for `mode`.  Optional:
 * gar_plan_prepare and the first Allreduce compile on demand. */
GAR_API int gar_plan_compile(gar_plan *plan, int mode);

/* Compiles and loads everything `mode` needs on the current device and uploads the
 * device tables.  Call before capturing Allreduce calls into a CUDA graph. */
GAR_API int gar_plan_prepare(gar_plan *plan, int mode);

/* The Allreduce (MPI_Allreduce with MPI_IN_PLACE, Sec. "Introduction").
 * rank_buffers: host array of P device pointers, each to n elements of the plan's
 * type, 16-byte aligned and pairwise distinct.  On return the work is enqueued on
 * `stream`; when it completes every buffer holds the reduction.  Rank x's block b is
 * the value at placement (x - b) mod P (x XOR b in the XOR group) after the paper's
 * schedule; for plans with one result copy (K = 1: bandwidth-optimal, fold and Ring
 * schedules) all ranks get identical bits, otherwise floating-point sums may differ in
 * the last bits between ranks (each rank's association order is a rotation of the same
 * tree).  The modes give identical bits. */
GAR_API int gar_allreduce(gar_plan *plan, void *const *rank_buffers, int mode, gar_stream_t stream);
/* The plan is not const in gar_allreduce, gar_allreduce_host and gar_allreduce_batched:
 * the first call on a device compiles and loads the plan's kernels, uploads its tables
 * and records the stream and step counts it ran with -- state that gar_plan_status and
 * gar_last_step_bytes read; the schedule itself never changes.
 * In GAR_STEP_PERSISTENT mode the return value only says that the launch was enqueued:
 * the results are complete only once gar_plan_status returns GAR_OK for the call. */

/* Host-buffer Allreduce: the P inputs host_in[x] are in host memory and the P results
 * go to host memory host_out[x] (host_out[x] may equal host_in[x], or another rank's
 * host_in; other overlaps are undefined).
 * GAR_FUSED with 16-byte-aligned host buffers that the GPU can address directly (pinned
 * or registered memory, or any host memory on a system with coherent host access such
 * as NVLink-C2C): one fused kernel reads the inputs from and writes the results to host
 * memory itself; dev_bufs is not used and may be NULL.  Otherwise the inputs are copied
 * (cudaMemcpyAsync per rank and element chunk) to dev_bufs -- P device buffers as for
 * gar_allreduce -- reduced there, and copied back; in fused mode the chunks pipeline
 * over internal streams that are forked from and joined back into `stream`.
 * Returns after enqueueing; synchronize the stream before reading host_out. */
GAR_API int gar_allreduce_host(gar_plan *plan, const void *const *host_in, void *const *host_out,
                       void *const *dev_bufs, int mode, gar_stream_t stream);

/* One instance of a batched Allreduce: `in` and `out` point to row-major [P][n]
 * arrays (rank x's vector is row x) for plans[plan]; in == out is allowed. */
typedef struct {
  int32_t plan;
  int32_t reserved;
  const void *in;
  void *out;
} gar_batch_desc;

/* Many independent small Allreduces in one fused launch (the 425-byte Allreduce of
 * Sec. "Introduction").  plans: nplans plans sharing dtype, op and n.  desc: DEVICE
 * array of `count` descriptors.  Instances whose pointers are not aligned for the
 * kernel's vector width fall back to element-wise loads inside the same kernel. */
GAR_API int gar_allreduce_batched(gar_plan *const *plans, int nplans, const gar_batch_desc *desc,
                          int count, gar_stream_t stream);

/* Outcome of the plan's most recent GAR_STEP_PERSISTENT Allreduce (no counterpart in
 * the paper: failure reporting of the bounded waits): waits for the stream it ran on,
 * then returns GAR_OK, GAR_ETIMEOUT if a grid-barrier wait gave up (the results are then
 * incomplete), or GAR_ECUDA.  GAR_OK if no persistent call ran. */
GAR_API int gar_plan_status(gar_plan *plan);

/* Barrier parameters of GAR_STEP_PERSISTENT (no counterpart in the paper).  spin_limit: polls (each an L2 round trip,
 * after the first 32 plus a 32 ns sleep) a CTA makes at a grid barrier before it gives up (0 restores the
 * default: 2^20 polls, roughly a second, or one poll per 256 bytes of memory traffic of
 * the plan's largest step if that is more -- a wait then outlasts that step many times
 * over).
 * phantom: extra arrivals the barrier waits for beyond the launched CTAs -- nonzero
 * values make every wait run out, which tests the timeout path without faulting
 * anything; keep 0 otherwise. */
GAR_API int gar_plan_debug_barrier(gar_plan *plan, unsigned int phantom, unsigned int spin_limit);

/* Bytes each communication step of the most recent step-faithful Allreduce read from
 * partner ranks, as counted by the kernels (S entries): the measured counterpart of the
 * per-step message volume of gar_plan_bytes (Sec. "Communication operator"); the
 * counting itself has no counterpart in the paper.  Synchronizes with the stream of
 * that call; GAR_ESTATE if no step-faithful call ran. */
GAR_API int gar_last_step_bytes(const gar_plan *plan, uint64_t *per_step);

/* Name of a GAR_* status code (static string).  Error reporting; no counterpart in the
 * paper. */
GAR_API const char *gar_strerror(int status);
/* The calling thread's most recent error detail (valid until its next failing call). */
GAR_API const char *gar_last_error(void);

/* The paper's cost model (Sec. "Communication model": tau = alpha + beta m + gamma m per
 * message, blocks of u = m / P bytes) for the version with S = steps:
 *   S = 2L (r = 0):      eq. bo_cost           2L alpha + 2(P-1) u beta + (P-1) u gamma
 *   L < S < 2L:          eq. intemediate_cost  (2L-r) alpha + (2(P-1) + (2^r-1)(L-1)) u beta
 *                                              + ((P-1) + (2^r-1)(2L-2)) u gamma
 *   S = L (r = L):       eq. lo_cost           L alpha + P L u beta + P (2L-2) u gamma
 * with L = ceil(log2 P), r = 2L - S, m_bytes = bytes per rank; beyond 2L:
 *   GAR_STEPS_RING:      eq. naive_cost        2(P-1) alpha + 2(P-1) u beta + (P-1) u gamma
 *   fold schedule, even S in (2L, 2(P-1)]:     S alpha + 2(P-1) u beta + (P-1) u gamma
 *     (the bandwidth-optimal traffic and combines in S steps; it equals eq. bo_cost at
 *     S = 2L and eq. naive_cost at S = 2(P-1)).
 * steps may be GAR_STEPS_BO / GAR_STEPS_LO.  Host-only.  Returns GAR_EINVAL for P < 1
 * or a step count the plans do not take. */
GAR_API int gar_cost_model(int P, int steps, double m_bytes, double alpha, double beta,
                           double gamma, double *tau);

/* The step count minimising gar_cost_model over the integers S in [L, 2L] (eq.
 * opt_number_of_steps gives the continuous optimum in log P; the library takes the
 * integer argmin, smallest S on ties).  Longer schedules are never cheaper in this model
 * (same traffic as S = 2L, more alpha terms).  Host-only. */
GAR_API int gar_optimal_steps(int P, double m_bytes, double alpha, double beta, double gamma,
                              int *steps);

/* Step-faithful Allreduce that allocates no device memory (cyclic-group plans only).  The paper has no
 * counterpart; this entry point serves callers that cannot call cudaMalloc when they
 * run an Allreduce, e.g. code whose device memory is all owned by a caching
 * allocator or by another runtime.  Same result as gar_allreduce(plan, rank_buffers,
 * GAR_STEP_FAITHFUL, stream), but the workspace is a fixed file-scope device array of
 * GAR_NOALLOC_SCRATCH_BYTES and the block ops travel in the kernel parameters; the
 * plan's workspace and device tables are not used, no bytes are recorded, and no
 * cudaMalloc, cudaFree or other allocating call is made.
 * The array exists on a device once the library's step kernels are loaded there; CUDA
 * loads them lazily: at the first step-faithful or persistent Allreduce, at
 * gar_plan_prepare(plan, GAR_STEP_FAITHFUL or GAR_STEP_PERSISTENT), or at the first call
 * of this function.  A caller whose allocator later takes all free memory should do one
 * of these first; the array then stays until the process exits.
 * Limits: P <= GAR_NOALLOC_MAX_P and a workspace (gar_plan_bytes) of at most
 * GAR_NOALLOC_SCRATCH_BYTES; larger plans return GAR_EINVAL with the sizes in
 * gar_last_error().  Every call looks up the array's address on the current device
 * (cudaGetSymbolAddress, which allocates nothing); make the first call on a device, or
 * the gar_plan_prepare above, before any stream capture.  All calls share the one array
 * and leave their partial results in it: calls whose work overlaps on the GPU (other
 * streams, other host threads) race, so order them on one stream.  rank_buffers: as for
 * gar_allreduce. */
#define GAR_NOALLOC_SCRATCH_BYTES (64u << 20)
#define GAR_NOALLOC_MAX_P 64
GAR_API int gar_allreduce_noalloc(gar_plan *plan, void *const *rank_buffers, gar_stream_t stream);

/* Library self-test for build checks: generates and compiles (host-only, no GPU) the
 * fused kernels of a few plans.  Returns GAR_OK or GAR_EJIT. */
GAR_API int gar_selftest_compile(void);

#ifdef __cplusplus
}
#endif

#endif /* GAR_H */
