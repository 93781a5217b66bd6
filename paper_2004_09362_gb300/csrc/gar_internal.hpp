// Internal definitions shared by the schedule builder, the code generator, the
// kernels and the C ABI.  Not part of the public interface (include/gar.h).
#pragma once

#include <cstdint>
#include <cstddef>
#include <string>
#include <vector>

#include "../../include/gar.h"

namespace gar {

// Buffers a step-faithful op reads or writes, per rank.
enum Buf : uint8_t {
  BUF_NONE = 0,
  BUF_RANK = 1,  // the caller's rank buffer (input, then output), element type T
  BUF_QP0 = 2,   // q' slots, ping (accumulation type)
  BUF_QP1 = 3,   // q' slots, pong
  BUF_QS = 4     // q* slots (accumulation type)
};
constexpr int NUM_WS_BUFS = 3;  // QP0, QP1, QS
// Each communication step's byte counter is spread over this many device slots (warps
// add to slot (global warp index mod STEP_BYTE_SLOTS)); the reader sums them.  One
// shared counter serialised ~10^5 same-address atomics per launch at L2.
constexpr int STEP_BYTE_SLOTS = 32;

// One block operation of a step-faithful launch, identical for every rank x.  With
// b = (x - dst_place) mod P (the block index, which a move never changes):
//   recv  = buf[recv_buf][(x + partner) mod P][block b]          (if recv_place >= 0)
//   out_k = own(buf[out_k_own][x][block b]) (+) recv  ->  buf[out_k_buf][x][block b]
// A missing own operand makes out_k a copy of recv; a missing recv a copy of own.
struct StepOp {
  int16_t recv_place;  // placement of the received vector at the partner, -1 = none
  int16_t dst_place;   // placement at this rank
  uint8_t recv_buf;
  uint8_t out0_buf, out0_own;
  uint8_t out1_buf, out1_own;
  uint8_t pad[7];
};
static_assert(sizeof(StepOp) == 16, "StepOp must stay 16 bytes");

struct Launch {
  int phase;         // 0 reduction step, 1 distribution step, 2 local finalize copy
  int comm_step;     // index of the communication step it implements, -1 for local
  int partner;       // rank x receives from (x + partner) mod P
  int first_op;      // into Plan::ops
  int nops;
};

// Launch descriptor as the persistent kernel reads it from device memory.
struct LaunchDesc {
  int first_op, nops, partner, comm_step;
};

struct CommStep {
  int phase;                      // 0 reduce, 1 distribute
  int i;                          // the paper's step index i
  int N, d;
  int partner;                    // cyclic: rank x receives from x + partner; XOR: x ^ partner
  std::vector<int32_t> tx;        // placements transmitted by every rank
  uint64_t msg_bytes;             // predicted, all ranks together
};

// Per-element-position program of the fused mode.
struct FusedProgram {
  int P = 0, K = 0;
  std::vector<int32_t> a, b;      // combine k: value P + k = a[k] (+) b[k]
  std::vector<int32_t> place;     // combine k: placement its result lives at (contribution j: j)
  std::vector<int8_t> star;       // combine k: 1 if its result is a q* vector, 0 if a q' vector
  std::vector<int32_t> out;       // out[s] = value id of result copy s
  std::vector<int32_t> origin;    // origin[p] = copy written to placement p
};

struct JitKernel;  // jit.cpp

constexpr int GAR_HOST_CHUNKS_MAX = 16;  // element chunks of the pipelined host path

}  // namespace gar

struct gar_plan {
  int P = 0, L = 0, S = 0, r = 0, K = 0;
  int group = 0;                  // GAR_GROUP_CYCLIC or GAR_GROUP_XOR
  bool ring = false;              // the Ring schedule (S = 2(P-1)) instead of S in [L, 2L]
  std::vector<int> folds;         // fold schedule (S > 2L): vectors folded per reduction step
  uint64_t n = 0;
  int dtype = 0, op = 0;
  uint64_t q = 0, rem = 0;        // block i has q + (i < rem) elements
  std::vector<int> N;             // N_0..N_L
  std::vector<gar::CommStep> comm;
  std::vector<gar::StepOp> ops;
  std::vector<gar::Launch> launches;
  bool ws_used[gar::NUM_WS_BUFS] = {false, false, false};
  uint64_t n_pad = 0;             // per-rank stride of workspace slices (elements)
  size_t ws_bytes = 0;
  gar::FusedProgram prog;

  // device state
  void *ws = nullptr;
  size_t ws_set_bytes = 0;
  int device = -1;
  gar::StepOp *d_ops = nullptr;
  unsigned long long *d_step_bytes = nullptr;
  gar_stream_t last_stream = nullptr;
  bool ran_step_faithful = false;
  gar::JitKernel *fused = nullptr;   // owned by the JIT cache
  int fused_width = 0;
  // persistent step-faithful mode: launch table, barrier state, barrier parameters
  void *d_launches = nullptr;
  void *d_barrier = nullptr;
  unsigned int barrier_spin_limit = 1u << 20;   // polls (each an L2 round trip); see default_spin_limit
  unsigned int barrier_phantom = 0;
  bool ran_persistent = false;
  // pipelined host-buffer path: 3 streams (to device, kernel, to host) and events
  bool hp_ready = false;
  void *hp_stream[3] = {nullptr, nullptr, nullptr};
  void *hp_h2d[gar::GAR_HOST_CHUNKS_MAX] = {};
  void *hp_krn[gar::GAR_HOST_CHUNKS_MAX] = {};
  void *hp_start = nullptr, *hp_done = nullptr;
};

namespace gar {

int elem_size(int dtype);
int acc_size(int dtype);
int ceil_log2(int P);

// plan.cpp
int build_plan(gar_plan *pl);

// codegen.cpp
struct CodegenResult {
  std::string source;
  std::string kernel_name;
  int width = 1;
  int table_copies = 1;  // fused kernels: copies of the in[] / out[] pointer tables (1 or 2)
  int threads = 256;     // threads per CTA
  int form = 0;          // fused kernels: 0 single-thread program, 1 breadth-first
};
// threads / minb > 0 override the CTA size and the minimum resident CTAs per SM
CodegenResult generate_fused_source(const gar_plan &pl, int threads = 0, int minb = 0, int fadd2 = -1);
// The breadth-first form of the fused kernel (programs with many result copies), and
// the peak number of live values of a plan's program in the single-thread form.
CodegenResult generate_fused_bf_source(const gar_plan &pl);
// two lanes per element position for rotation-invariant (latency-optimal cyclic) programs
bool split_form_applies(const gar_plan &pl);
CodegenResult generate_fused_split_source(const gar_plan &pl);
int fused_peak_live(const gar_plan &pl);
CodegenResult generate_batched_source(const std::vector<const gar_plan *> &plans);

// jit.cpp
struct JitKernel {
  void *library = nullptr;   // cudaLibrary_t
  void *kernel = nullptr;    // cudaKernel_t
  std::vector<char> cubin;
  std::string source;        // the generated CUDA source it was compiled from
  std::string name;
  int width = 1;
  int table_copies = 1;
  int threads = 256;
  int form = 0;
  int blocks_per_sm = 0;
  int regs = 0, local_bytes = 0;
  bool loaded = false;
};
int jit_compile(const CodegenResult &cg, JitKernel **out);
int jit_load(JitKernel *k);

// step_kernels.cu
int launch_step(const gar_plan &pl, const Launch &ln, int launch_index, void *const *rank,
                gar_stream_t stream);
int launch_persistent(const gar_plan &pl, void *const *rank, gar_stream_t stream);
size_t barrier_state_bytes();
int load_step_module();

// api.cpp
void set_error(const std::string &msg);
const char *last_error_cstr();
int cuda_fail(int err, const char *what);

}  // namespace gar
