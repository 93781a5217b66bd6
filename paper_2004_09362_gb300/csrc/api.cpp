// C ABI of the permutation-group Allreduce library (declared in include/gar.h).
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <new>
#include <stdexcept>
#include <string>
#include <vector>

#include "gar_internal.hpp"

namespace gar {

namespace {
thread_local std::string t_last_error;
}

void set_error(const std::string &msg) { t_last_error = msg; }
const char *last_error_cstr() { return t_last_error.c_str(); }

int cuda_fail(int err, const char *what) {
  set_error(std::string(what) + ": " + cudaGetErrorString((cudaError_t)err));
  return GAR_ECUDA;
}

namespace {

int check_plan(const gar_plan *pl) {
  if (pl == nullptr) {
    set_error("null plan");
    return GAR_EINVAL;
  }
  return GAR_OK;
}

int check_mode(int mode) {
  if (mode != GAR_STEP_FAITHFUL && mode != GAR_FUSED && mode != GAR_STEP_PERSISTENT) {
    set_error("unknown mode");
    return GAR_EINVAL;
  }
  return GAR_OK;
}

int ensure_device(gar_plan *pl) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (pl->device >= 0 && pl->device != dev) {
    set_error("plan was prepared on another device");
    return GAR_ESTATE;
  }
  pl->device = dev;
  return GAR_OK;
}

// Default poll limit of the persistent kernel's grid barriers: 2^20 polls (about a
// second), or one poll per 256 bytes that the plan's largest step reads and writes (a
// combine step: partner read, own read, write -- at most 3x its message bytes), so that
// a legitimate wait never runs out however large the vectors are.
unsigned int default_spin_limit(const gar_plan &pl) {
  uint64_t most = 0;
  for (const CommStep &cs : pl.comm) most = std::max<uint64_t>(most, 3 * cs.msg_bytes);
  const uint64_t polls = std::max<uint64_t>(1u << 20, most / 256);
  return (unsigned int)std::min<uint64_t>(polls, 0xffffffffull);
}

int prepare_step_faithful(gar_plan *pl) {
  int rc = ensure_device(pl);
  if (rc) return rc;
  // the step kernels' module, loaded now rather than at the first launch
  if ((rc = load_step_module())) return rc;
  if (pl->d_ops == nullptr && !pl->ops.empty()) {
    cudaError_t e = cudaMalloc(&pl->d_ops, pl->ops.size() * sizeof(StepOp));
    if (e != cudaSuccess) return cuda_fail(e, "cudaMalloc(op table)");
    e = cudaMemcpy(pl->d_ops, pl->ops.data(), pl->ops.size() * sizeof(StepOp),
                   cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy(op table)");
  }
  if (pl->d_launches == nullptr && !pl->launches.empty()) {
    std::vector<LaunchDesc> ld;
    for (const Launch &ln : pl->launches) ld.push_back({ln.first_op, ln.nops, ln.partner, ln.comm_step});
    cudaError_t e = cudaMalloc(&pl->d_launches, ld.size() * sizeof(LaunchDesc));
    if (e != cudaSuccess) return cuda_fail(e, "cudaMalloc(launch table)");
    e = cudaMemcpy(pl->d_launches, ld.data(), ld.size() * sizeof(LaunchDesc), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy(launch table)");
  }
  if (pl->d_barrier == nullptr) {
    cudaError_t e = cudaMalloc(&pl->d_barrier, barrier_state_bytes());
    if (e != cudaSuccess) return cuda_fail(e, "cudaMalloc(barrier state)");
    e = cudaMemset(pl->d_barrier, 0, barrier_state_bytes());
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemset(barrier state)");
  }
  if (pl->d_step_bytes == nullptr && pl->S > 0) {
    const size_t cbytes = (size_t)pl->S * STEP_BYTE_SLOTS * sizeof(unsigned long long);
    cudaError_t e = cudaMalloc(&pl->d_step_bytes, cbytes);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMalloc(step counters)");
    e = cudaMemset(pl->d_step_bytes, 0, cbytes);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemset(step counters)");
  }
  return GAR_OK;
}

// Fused mode compiles the plan's program as straight-line code; the compile time grows
// faster than linearly with its size (P = 300, 3900 operations: about a minute).
int check_fused_size(const gar_plan *pl) {
  const size_t ops = pl->prog.a.size() + 2 * (size_t)pl->P;
  if (ops > GAR_FUSED_MAX_OPS) {
    set_error("fused program of " + std::to_string(ops) + " operations (" +
              std::to_string(pl->prog.a.size()) + " combines + " + std::to_string(2 * pl->P) +
              " loads and stores) exceeds GAR_FUSED_MAX_OPS = " + std::to_string(GAR_FUSED_MAX_OPS) +
              "; use GAR_STEP_FAITHFUL");
    return GAR_EINVAL;
  }
  return GAR_OK;
}

// The fused kernel a plan uses.  Float sums with several result copies whose
// single-thread program keeps more than 160 values alive per element position (P = 127
// at S = 7 and 8: 254 and 192) are register-bound in that form and take the
// breadth-first form (0.59 instead of 0.68 ms, and 0.47 instead of 0.56 ms, at P = 127 x
// 8 MiB bf16 on GB300); every other plan takes the single-thread form.  GAR_TUNE_FUSED_FORM
// (0, 1 or 2) forces one form, for parity tests and launch-shape sweeps; the two-lane
// form (2) exists for latency-optimal cyclic programs only and is never the default (P =
// 127 x 8 MiB bf16 S = 7: 0.78 ms against 0.60 ms breadth-first in one pass, 0.55 ms in
// two; fp32: 0.416 against 0.409 ms in one pass).
int fused_form(const gar_plan &pl) {
  if (pl.K <= 1) return GAR_FORM_SINGLE;
  const char *ff = std::getenv("GAR_TUNE_FUSED_FORM");
  if (ff && *ff) {
    const int f = std::atoi(ff);
    if (f == GAR_FORM_SPLIT) return split_form_applies(pl) ? GAR_FORM_SPLIT : GAR_FORM_BREADTH;
    return f == GAR_FORM_BREADTH ? GAR_FORM_BREADTH : GAR_FORM_SINGLE;
  }
  return (pl.op == GAR_SUM && pl.dtype != GAR_I32 && fused_peak_live(pl) > 160) ? GAR_FORM_BREADTH
                                                                                : GAR_FORM_SINGLE;
}

CodegenResult fused_codegen(const gar_plan &pl) {
  switch (fused_form(pl)) {
    case GAR_FORM_BREADTH: return generate_fused_bf_source(pl);
    case GAR_FORM_SPLIT: return generate_fused_split_source(pl);
    default: return generate_fused_source(pl);
  }
}

int compile_fused(gar_plan *pl) {
  if (pl->fused) return GAR_OK;
  if (int rc = check_fused_size(pl)) return rc;
  CodegenResult cg;
  try {
    cg = fused_codegen(*pl);
  } catch (const std::exception &ex) {
    set_error(std::string("fused code generation: ") + ex.what());
    return GAR_EINVAL;
  }
  JitKernel *k = nullptr;
  int rc = jit_compile(cg, &k);
  if (rc) return rc;
  pl->fused = k;
  pl->fused_width = k->width;
  return GAR_OK;
}

// Register-heavy single-thread kernels (more than 128 registers once loaded) run in
// 64-thread CTAs capped at 168 registers, so that three warps share each sub-partition's
// register file and the small CTAs of an SM drift apart.  On GB300: P = 32 x 32 MiB bf16
// latency-optimal (208 registers) 0.426 -> 0.338 ms; P = 127 x 8 MiB bf16 S = 9 (200)
// 0.434 -> 0.401 ms, S = 11 (174) 0.344 -> 0.324 ms; kernels at 128 registers or fewer
// were unchanged or slower (P = 64 fp32 latency-optimal, 40 registers: 0.33 -> 0.40 ms).
// When the 168-register build spills more than 256 bytes per thread, 32-thread CTAs with
// the full 255 registers (two warps per sub-partition) are built too and kept if they
// spill less: P = 127 x 8 MiB bf16 S = 10 (168 registers + 328 B spilled, 0.369 ms;
// 250 registers, no spill, 0.351 ms).  Smaller spills cost less than the lost warps:
// P = 32 x 32 MiB bf16 S = 5 (152 B: 0.341 ms against 0.390 ms at 210 registers),
// P = 64 x 16 MiB bf16 S = 8 (96 B: 0.324 against 0.346), P = 127 S = 9 (48 B: 0.407
// against 0.460).
// The counts are the loaded kernel's own (the compiler's log does not always carry them).
int prepare_fused(gar_plan *pl) {
  int rc = compile_fused(pl);
  if (rc) return rc;
  rc = ensure_device(pl);
  if (rc) return rc;
  if ((rc = jit_load(pl->fused))) return rc;
  const bool shape_forced = std::getenv("GAR_TUNE_FUSED_THREADS") || std::getenv("GAR_TUNE_FUSED_MINB");
  if (pl->fused->form != 0 || pl->fused->threads != 256 || shape_forced || pl->fused->regs <= 128)
    return GAR_OK;
  auto build = [&](int threads, int minb, int fadd2, JitKernel **out) -> int {
    CodegenResult cg;
    try {
      cg = generate_fused_source(*pl, threads, minb, fadd2);
    } catch (const std::exception &ex) {
      set_error(std::string("fused code generation: ") + ex.what());
      return GAR_EINVAL;
    }
    if (int r = jit_compile(cg, out)) return r;
    return jit_load(*out);
  };
  JitKernel *k = nullptr;
  if ((rc = build(64, 5, -1, &k))) return rc;
  if (k->local_bytes > 256) {
    JitKernel *wide = nullptr;
    if ((rc = build(32, 8, -1, &wide))) return rc;
    if (wide->local_bytes < k->local_bytes) k = wide;
  }
  // bf16 kernels of 2-element vectors take paired fp32 adds only when the capped build is
  // register-bound anyway (at the cap and spilling) and the paired build spills no more:
  // then the pairs halve the adds at no cost in warps (P = 127 x 8 MiB S = 9: 0.405 ->
  // 0.372 ms).  Elsewhere they cost registers: P = 100 S = 9 (128 -> 140 registers) 0.272
  // -> 0.280 ms, P = 64 latency-optimal (39 -> 255) 0.339 -> 0.493 ms.
  if (pl->dtype == GAR_BF16 && k->width == 2 && k->local_bytes > 0 && k->regs >= 168 &&
      !std::getenv("GAR_TUNE_FADD2")) {
    JitKernel *paired = nullptr;
    if ((rc = build(k->threads, k->threads == 64 ? 5 : 8, 1, &paired))) return rc;
    if (paired->local_bytes <= k->local_bytes) k = paired;
  }
  pl->fused = k;
  pl->fused_width = k->width;
  return GAR_OK;
}

int check_buffers(const gar_plan *pl, void *const *bufs) {
  if (bufs == nullptr) {
    set_error("null rank buffer array");
    return GAR_EINVAL;
  }
  std::vector<uintptr_t> ptrs(pl->P);
  for (int x = 0; x < pl->P; ++x) {
    if (bufs[x] == nullptr) {
      set_error("null rank buffer " + std::to_string(x));
      return GAR_EINVAL;
    }
    if (reinterpret_cast<uintptr_t>(bufs[x]) % 16 != 0) {
      set_error("rank buffer " + std::to_string(x) + " is not 16-byte aligned");
      return GAR_EALIGN;
    }
    ptrs[x] = reinterpret_cast<uintptr_t>(bufs[x]);
  }
  std::sort(ptrs.begin(), ptrs.end());
  if (std::adjacent_find(ptrs.begin(), ptrs.end()) != ptrs.end()) {
    set_error("two ranks share one buffer");
    return GAR_EINVAL;
  }
  return GAR_OK;
}

int grid_for(const JitKernel *k, uint64_t work_items) {
  // One work item per thread: with many more CTAs than fit at once the block scheduler
  // keeps every SM full and each thread's loads are in flight together (a persistent
  // grid-stride loop serialises a thread's iterations and ran 6% slower on GB300).
  // GAR_TUNE_GRID_WAVES caps the grid at that many waves of resident CTAs (launch-shape
  // sweeps only); the kernels' grid-stride loops cover any remainder.
  const uint64_t need = (work_items + k->threads - 1) / k->threads;
  uint64_t cap = 0x7fffffffull;
  const char *wv = std::getenv("GAR_TUNE_GRID_WAVES");
  if (wv && std::atoi(wv) > 0) {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 1;
    cap = (uint64_t)sms * (uint64_t)std::max(1, k->blocks_per_sm) * (uint64_t)std::atoi(wv);
  }
  return (int)std::max<uint64_t>(1, std::min<uint64_t>(need, cap));
}

// Launches a generated kernel with programmatic stream serialisation: back-to-back
// calls overlap one launch's start with the previous one's drain.  Every generated
// kernel runs griddepcontrol.wait before its first read, so it still sees all the work
// of earlier kernels on the stream.
cudaError_t launch_generated(const JitKernel *k, int grid, void **kargs, gar_stream_t stream) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(k->threads);
  cfg.stream = (cudaStream_t)stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelExC(&cfg, (const void *)k->kernel, kargs);
}

// One fused launch over element positions [e_lo, e_hi) (e_lo a multiple of the
// kernel's vector width).  The parameter block is the generated kernel's gar_args:
// P input pointers, P output pointers, e_lo, e_hi.
int launch_fused_range(gar_plan *pl, const void *const *in, void *const *out, uint64_t e_lo,
                       uint64_t e_hi, gar_stream_t stream) {
  if (e_hi <= e_lo) return GAR_OK;
  // gar_args: the in[] table, then the out[] table, each table_copies times in a row,
  // then e_lo, e_hi
  const size_t pb = 8 * (size_t)pl->P;
  const int copies = pl->fused->table_copies;
  std::vector<unsigned char> args(2 * copies * pb + 16);
  unsigned char *w = args.data();
  for (int c = 0; c < copies; ++c, w += pb) std::memcpy(w, in, pb);
  for (int c = 0; c < copies; ++c, w += pb) std::memcpy(w, out, pb);
  std::memcpy(w, &e_lo, 8);
  std::memcpy(w + 8, &e_hi, 8);
  void *kargs[] = {args.data()};
  // threads: one per vector of `width` positions, or two per position in groups of 16
  // (two-lane form)
  const uint64_t items = pl->fused->form == GAR_FORM_SPLIT ? (e_hi - e_lo + 15) / 16 * 32
                                                           : (e_hi - e_lo) / pl->fused->width + 1;
  const int grid = grid_for(pl->fused, items);
  cudaError_t e = launch_generated(pl->fused, grid, kargs, stream);
  if (e != cudaSuccess) return cuda_fail(e, "fused kernel launch");
  return GAR_OK;
}

int run_fused(gar_plan *pl, void *const *rank, gar_stream_t stream) {
  int rc = prepare_fused(pl);
  if (rc) return rc;
  return launch_fused_range(pl, rank, rank, 0, pl->n, stream);
}

// True when every pointer is host memory the GPU can read and write directly (pinned or
// registered memory, or any host memory on a system with coherent access such as
// NVLink-C2C), so a kernel can use it without staging copies.
bool device_accessible_host(const void *const *ptrs, int count) {
  int dev = 0, pageable = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&pageable, cudaDevAttrPageableMemoryAccess, dev);
  for (int x = 0; x < count; ++x) {
    cudaPointerAttributes at{};
    if (cudaPointerGetAttributes(&at, ptrs[x]) != cudaSuccess) {
      cudaGetLastError();
      return false;
    }
    const bool pinned = at.type == cudaMemoryTypeHost && at.devicePointer == ptrs[x];
    const bool pageable_ok = at.type == cudaMemoryTypeUnregistered && pageable;
    if (!pinned && !pageable_ok) return false;
  }
  return true;
}

// Internal streams and events of the pipelined host-buffer path (created once).
int prepare_host_pipeline(gar_plan *pl) {
  if (pl->hp_ready) return GAR_OK;
  cudaError_t e = cudaSuccess;
  for (int k = 0; k < 3 && e == cudaSuccess; ++k)
    e = cudaStreamCreateWithFlags((cudaStream_t *)&pl->hp_stream[k], cudaStreamNonBlocking);
  for (int c = 0; c < GAR_HOST_CHUNKS_MAX && e == cudaSuccess; ++c) {
    e = cudaEventCreateWithFlags((cudaEvent_t *)&pl->hp_h2d[c], cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags((cudaEvent_t *)&pl->hp_krn[c], cudaEventDisableTiming);
  }
  if (e == cudaSuccess) e = cudaEventCreateWithFlags((cudaEvent_t *)&pl->hp_start, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags((cudaEvent_t *)&pl->hp_done, cudaEventDisableTiming);
  if (e != cudaSuccess) return cuda_fail(e, "creating host-pipeline streams/events");
  pl->hp_ready = true;
  return GAR_OK;
}

// Fused Allreduce of host buffers, pipelined over element chunks: the copy of chunk c
// to the device, the kernel on chunk c and the copy of chunk c back run on three
// streams, so both copy directions and the kernel overlap.  Every element position
// depends only on the P contributions at that position, so chunks are independent.
int run_host_pipelined(gar_plan *pl, const void *const *host_in, void *const *host_out,
                       void *const *dev, gar_stream_t stream) {
  int rc = prepare_fused(pl);
  if (rc) return rc;
  rc = prepare_host_pipeline(pl);
  if (rc) return rc;
  const size_t es = (size_t)elem_size(pl->dtype);
  const uint64_t n = pl->n;
  uint64_t chunk = (n + GAR_HOST_CHUNKS_MAX - 1) / GAR_HOST_CHUNKS_MAX;
  chunk = std::max<uint64_t>(chunk, (uint64_t)1 << 16);
  chunk = (chunk + 63) / 64 * 64;
  const int nchunks = (int)((n + chunk - 1) / chunk);
  cudaStream_t s_in = (cudaStream_t)pl->hp_stream[0], s_k = (cudaStream_t)pl->hp_stream[1],
               s_out = (cudaStream_t)pl->hp_stream[2];
  cudaError_t e = cudaEventRecord((cudaEvent_t)pl->hp_start, (cudaStream_t)stream);
  for (int k = 0; k < 3 && e == cudaSuccess; ++k)
    e = cudaStreamWaitEvent((cudaStream_t)pl->hp_stream[k], (cudaEvent_t)pl->hp_start, 0);
  if (e != cudaSuccess) return cuda_fail(e, "host pipeline: fork");
  for (int c = 0; c < nchunks; ++c) {
    const uint64_t lo = (uint64_t)c * chunk, hi = std::min<uint64_t>(n, lo + chunk);
    const size_t off = (size_t)lo * es, bytes = (size_t)(hi - lo) * es;
    for (int x = 0; x < pl->P && e == cudaSuccess; ++x)
      e = cudaMemcpyAsync(static_cast<char *>(dev[x]) + off, static_cast<const char *>(host_in[x]) + off,
                          bytes, cudaMemcpyHostToDevice, s_in);
    if (e == cudaSuccess) e = cudaEventRecord((cudaEvent_t)pl->hp_h2d[c], s_in);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s_k, (cudaEvent_t)pl->hp_h2d[c], 0);
    if (e != cudaSuccess) return cuda_fail(e, "host pipeline: host to device");
    rc = launch_fused_range(pl, dev, dev, lo, hi, (gar_stream_t)s_k);
    if (rc) return rc;
    e = cudaEventRecord((cudaEvent_t)pl->hp_krn[c], s_k);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s_out, (cudaEvent_t)pl->hp_krn[c], 0);
    for (int x = 0; x < pl->P && e == cudaSuccess; ++x)
      e = cudaMemcpyAsync(static_cast<char *>(host_out[x]) + off, static_cast<const char *>(dev[x]) + off,
                          bytes, cudaMemcpyDeviceToHost, s_out);
    if (e != cudaSuccess) return cuda_fail(e, "host pipeline: device to host");
  }
  e = cudaEventRecord((cudaEvent_t)pl->hp_done, s_out);
  if (e == cudaSuccess) e = cudaStreamWaitEvent((cudaStream_t)stream, (cudaEvent_t)pl->hp_done, 0);
  if (e != cudaSuccess) return cuda_fail(e, "host pipeline: join");
  return GAR_OK;
}

int run_step_faithful(gar_plan *pl, void *const *rank, gar_stream_t stream, bool persistent) {
  int rc = prepare_step_faithful(pl);
  if (rc) return rc;
  if (pl->ws_bytes > 0) {
    if (pl->ws == nullptr || pl->ws_set_bytes < pl->ws_bytes) {
      set_error("step-faithful mode needs a workspace of " + std::to_string(pl->ws_bytes) +
                " bytes (gar_plan_set_workspace)");
      return GAR_ENOWS;
    }
  }
  cudaError_t e = cudaMemsetAsync(pl->d_step_bytes, 0,
                                  (size_t)pl->S * STEP_BYTE_SLOTS * sizeof(unsigned long long),
                                  (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync(step counters)");
  if (persistent) {
    e = cudaMemsetAsync(pl->d_barrier, 0, barrier_state_bytes(), (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync(barrier state)");
    rc = launch_persistent(*pl, rank, stream);
    if (rc) return rc;
    pl->ran_persistent = true;
  } else {
    for (size_t li = 0; li < pl->launches.size(); ++li) {
      rc = launch_step(*pl, pl->launches[li], (int)li, rank, stream);
      if (rc) return rc;
    }
  }
  pl->last_stream = stream;
  pl->ran_step_faithful = true;
  return GAR_OK;
}

}  // namespace
}  // namespace gar

using namespace gar;

extern "C" {

int gar_plan_create(gar_plan **out, int P, uint64_t n, int dtype, int op, int steps) {
  return gar_plan_create_group(out, P, n, dtype, op, steps, GAR_GROUP_CYCLIC);
}

int gar_plan_create_group(gar_plan **out, int P, uint64_t n, int dtype, int op, int steps, int group) {
  if (out == nullptr) {
    set_error("null output pointer");
    return GAR_EINVAL;
  }
  if (P < 1 || P > GAR_MAX_P) {
    set_error("P must be in [1, " + std::to_string(GAR_MAX_P) + "]");
    return GAR_EINVAL;
  }
  if (dtype != GAR_F32 && dtype != GAR_BF16 && dtype != GAR_I32) {
    set_error("unknown dtype");
    return GAR_EINVAL;
  }
  if (op != GAR_SUM && op != GAR_MAX && op != GAR_MIN) {
    set_error("unknown op");
    return GAR_EINVAL;
  }
  if (n > (uint64_t)1 << 40) {
    set_error("n too large");
    return GAR_EINVAL;
  }
  if (group != GAR_GROUP_CYCLIC && group != GAR_GROUP_XOR) {
    set_error("unknown group");
    return GAR_EINVAL;
  }
  if (group == GAR_GROUP_XOR && (P & (P - 1)) != 0) {
    set_error("the XOR group needs P a power of two");
    return GAR_EINVAL;
  }
  const int L = ceil_log2(P);
  int S = steps;
  const bool ring = steps == GAR_STEPS_RING;
  if (ring && group != GAR_GROUP_CYCLIC) {
    set_error("the Ring schedule uses the cyclic group");
    return GAR_EINVAL;
  }
  if (steps == GAR_STEPS_BO) S = 2 * L;
  if (steps == GAR_STEPS_LO) S = L;
  if (ring) S = 2 * (P - 1);
  const bool folded = !ring && S > 2 * L && S <= 2 * (P - 1) && S % 2 == 0;
  if (folded && group != GAR_GROUP_CYCLIC) {
    set_error("step counts beyond 2L use the cyclic group");
    return GAR_EINVAL;
  }
  if (!ring && !folded && (S < L || S > 2 * L)) {
    set_error("steps must be in [" + std::to_string(L) + ", " + std::to_string(2 * L) +
              "] or even up to " + std::to_string(2 * (P - 1)) + " for P=" + std::to_string(P));
    return GAR_EINVAL;
  }
  gar_plan *pl = new (std::nothrow) gar_plan();
  if (pl == nullptr) return GAR_ENOMEM;
  pl->P = P;
  pl->n = n;
  pl->dtype = dtype;
  pl->op = op;
  pl->S = S;
  pl->group = group;
  pl->ring = ring;
  int rc = build_plan(pl);
  if (rc) {
    delete pl;
    return rc;
  }
  pl->barrier_spin_limit = default_spin_limit(*pl);
  *out = pl;
  return GAR_OK;
}

void gar_plan_destroy(gar_plan *pl) {
  if (pl == nullptr) return;
  if (pl->d_ops) cudaFree(pl->d_ops);
  if (pl->d_step_bytes) cudaFree(pl->d_step_bytes);
  if (pl->d_launches) cudaFree(pl->d_launches);
  if (pl->d_barrier) cudaFree(pl->d_barrier);
  if (pl->hp_ready) {
    for (int k = 0; k < 3; ++k) cudaStreamDestroy((cudaStream_t)pl->hp_stream[k]);
    for (int c = 0; c < GAR_HOST_CHUNKS_MAX; ++c) {
      cudaEventDestroy((cudaEvent_t)pl->hp_h2d[c]);
      cudaEventDestroy((cudaEvent_t)pl->hp_krn[c]);
    }
    cudaEventDestroy((cudaEvent_t)pl->hp_start);
    cudaEventDestroy((cudaEvent_t)pl->hp_done);
  }
  delete pl;
}

int gar_plan_get_info(const gar_plan *pl, gar_plan_info *info) {
  if (int rc = check_plan(pl)) return rc;
  if (info == nullptr) return GAR_EINVAL;
  std::memset(info, 0, sizeof *info);
  info->P = pl->P;
  info->L = pl->L;
  info->S = pl->S;
  info->r = pl->r;
  info->K = pl->K;
  info->dtype = pl->dtype;
  info->op = pl->op;
  info->n_launches = (int)pl->launches.size();
  info->n = pl->n;
  info->fused_combines = (int)pl->prog.a.size();
  info->group = pl->group;
  info->ring = pl->ring ? 1 : 0;
  info->fused_form = pl->fused != nullptr ? pl->fused->form : fused_form(*pl);
  info->fused_width = pl->fused_width;
  if (pl->fused != nullptr && pl->fused->loaded) {
    info->fused_regs = pl->fused->regs;
    info->fused_local_bytes = pl->fused->local_bytes;
  }
  return GAR_OK;
}

int gar_plan_bytes(const gar_plan *pl, size_t *workspace_bytes, uint64_t *msg_bytes_per_step, int *S) {
  if (int rc = check_plan(pl)) return rc;
  if (workspace_bytes) *workspace_bytes = pl->ws_bytes;
  if (msg_bytes_per_step)
    for (int t = 0; t < pl->S; ++t) msg_bytes_per_step[t] = pl->comm[t].msg_bytes;
  if (S) *S = pl->S;
  return GAR_OK;
}

int gar_plan_step(const gar_plan *pl, int t, int *phase, int *partner, int32_t *placements, int *count) {
  if (int rc = check_plan(pl)) return rc;
  if (t < 0 || t >= pl->S) {
    set_error("step index out of range");
    return GAR_EINVAL;
  }
  const CommStep &cs = pl->comm[t];
  if (phase) *phase = cs.phase;
  if (partner) *partner = cs.partner;
  if (count) *count = (int)cs.tx.size();
  if (placements) std::copy(cs.tx.begin(), cs.tx.end(), placements);
  return GAR_OK;
}

int gar_plan_origin(const gar_plan *pl, int32_t *origin) {
  if (int rc = check_plan(pl)) return rc;
  if (origin == nullptr) return GAR_EINVAL;
  std::copy(pl->prog.origin.begin(), pl->prog.origin.end(), origin);
  return GAR_OK;
}

int gar_plan_fused_program(const gar_plan *pl, int32_t *ops, int *nops, int32_t *outputs) {
  if (int rc = check_plan(pl)) return rc;
  if (nops == nullptr) return GAR_EINVAL;
  *nops = (int)pl->prog.a.size();
  if (ops)
    for (size_t k = 0; k < pl->prog.a.size(); ++k) {
      ops[2 * k] = pl->prog.a[k];
      ops[2 * k + 1] = pl->prog.b[k];
    }
  if (outputs) std::copy(pl->prog.out.begin(), pl->prog.out.end(), outputs);
  return GAR_OK;
}

int gar_plan_step_ops(const gar_plan *pl, int32_t *ops, int *nops, int32_t *launch_partner, int *nlaunch) {
  if (int rc = check_plan(pl)) return rc;
  if (nops) *nops = (int)pl->ops.size();
  if (nlaunch) *nlaunch = (int)pl->launches.size();
  if (launch_partner)
    for (size_t l = 0; l < pl->launches.size(); ++l) launch_partner[l] = pl->launches[l].partner;
  if (ops) {
    for (size_t l = 0; l < pl->launches.size(); ++l) {
      const Launch &ln = pl->launches[l];
      for (int k = 0; k < ln.nops; ++k) {
        const StepOp &op = pl->ops[ln.first_op + k];
        int32_t *o = ops + 8 * (size_t)(ln.first_op + k);
        o[0] = (int32_t)l;
        o[1] = op.recv_place;
        o[2] = op.dst_place;
        o[3] = op.recv_buf;
        o[4] = op.out0_buf;
        o[5] = op.out0_own;
        o[6] = op.out1_buf;
        o[7] = op.out1_own;
      }
    }
  }
  return GAR_OK;
}

int gar_plan_fused_source(const gar_plan *pl, char *buf, size_t *len) {
  if (int rc = check_plan(pl)) return rc;
  if (len == nullptr) return GAR_EINVAL;
  std::string src;
  try {
    src = pl->fused != nullptr ? pl->fused->source : fused_codegen(*pl).source;
  } catch (const std::exception &ex) {
    set_error(std::string("fused code generation: ") + ex.what());
    return GAR_EINVAL;
  }
  if (buf != nullptr && *len > 0) {
    const size_t m = std::min(*len - 1, src.size());
    std::memcpy(buf, src.data(), m);
    buf[m] = '\0';
  }
  *len = src.size() + 1;
  return GAR_OK;
}

int gar_plan_set_workspace(gar_plan *pl, void *dev_ptr, size_t bytes) {
  if (int rc = check_plan(pl)) return rc;
  if (dev_ptr == nullptr && bytes != 0) return GAR_EINVAL;
  if (reinterpret_cast<uintptr_t>(dev_ptr) % 16 != 0) {
    set_error("workspace is not 16-byte aligned");
    return GAR_EALIGN;
  }
  pl->ws = dev_ptr;
  pl->ws_set_bytes = bytes;
  return GAR_OK;
}

int gar_plan_compile(gar_plan *pl, int mode) {
  if (int rc = check_plan(pl)) return rc;
  if (int rc = check_mode(mode)) return rc;
  if (mode == GAR_FUSED) return compile_fused(pl);
  return GAR_OK;
}

int gar_plan_prepare(gar_plan *pl, int mode) {
  if (int rc = check_plan(pl)) return rc;
  if (int rc = check_mode(mode)) return rc;
  if (mode == GAR_FUSED) return prepare_fused(pl);
  return prepare_step_faithful(pl);
}

int gar_allreduce(gar_plan *pl, void *const *rank_buffers, int mode, gar_stream_t stream) {
  if (int rc = check_plan(pl)) return rc;
  if (int rc = check_mode(mode)) return rc;
  if (int rc = check_buffers(pl, rank_buffers)) return rc;
  if (pl->n == 0 || pl->P == 1) return GAR_OK;
  if (mode == GAR_FUSED) return run_fused(pl, rank_buffers, stream);
  return run_step_faithful(pl, rank_buffers, stream, mode == GAR_STEP_PERSISTENT);
}

int gar_allreduce_host(gar_plan *pl, const void *const *host_in, void *const *host_out,
                       void *const *dev_bufs, int mode, gar_stream_t stream) {
  if (int rc = check_plan(pl)) return rc;
  if (int rc = check_mode(mode)) return rc;
  if (host_in == nullptr || host_out == nullptr) {
    set_error("null host buffer array");
    return GAR_EINVAL;
  }
  for (int x = 0; x < pl->P; ++x) {
    if (host_in[x] == nullptr || host_out[x] == nullptr) {
      set_error("null host buffer");
      return GAR_EINVAL;
    }
  }
  if (pl->n == 0) return GAR_OK;
  const size_t bytes = (size_t)pl->n * (size_t)elem_size(pl->dtype);
  if (mode == GAR_FUSED && pl->P > 1) {
    bool aligned = true;
    for (int x = 0; x < pl->P; ++x)
      aligned = aligned && reinterpret_cast<uintptr_t>(host_in[x]) % 16 == 0 &&
                reinterpret_cast<uintptr_t>(host_out[x]) % 16 == 0;
    if (aligned && device_accessible_host(host_in, pl->P) &&
        device_accessible_host(reinterpret_cast<const void *const *>(host_out), pl->P)) {
      // The kernel reads the inputs from and writes the results to host memory itself.
      int rc = prepare_fused(pl);
      if (rc) return rc;
      return launch_fused_range(pl, host_in, host_out, 0, pl->n, stream);
    }
    if (int rc = check_buffers(pl, dev_bufs)) return rc;
    return run_host_pipelined(pl, host_in, host_out, dev_bufs, stream);
  }
  if (int rc = check_buffers(pl, dev_bufs)) return rc;
  for (int x = 0; x < pl->P && bytes; ++x) {
    cudaError_t e = cudaMemcpyAsync(dev_bufs[x], host_in[x], bytes, cudaMemcpyHostToDevice,
                                    (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync(host to device)");
  }
  int rc = gar_allreduce(pl, dev_bufs, mode, stream);
  if (rc) return rc;
  for (int x = 0; x < pl->P && bytes; ++x) {
    cudaError_t e = cudaMemcpyAsync(host_out[x], dev_bufs[x], bytes, cudaMemcpyDeviceToHost,
                                    (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync(device to host)");
  }
  return GAR_OK;
}

int gar_allreduce_batched(gar_plan *const *plans, int nplans, const gar_batch_desc *desc, int count,
                          gar_stream_t stream) {
  if (plans == nullptr || nplans < 1 || count < 0 || (count > 0 && desc == nullptr)) {
    set_error("bad batched arguments");
    return GAR_EINVAL;
  }
  std::vector<const gar_plan *> ps;
  for (int k = 0; k < nplans; ++k) {
    if (plans[k] == nullptr) {
      set_error("null plan in batch");
      return GAR_EINVAL;
    }
    if (plans[k]->dtype != plans[0]->dtype || plans[k]->op != plans[0]->op ||
        plans[k]->n != plans[0]->n) {
      set_error("batched plans must share dtype, op and n");
      return GAR_EINVAL;
    }
    ps.push_back(plans[k]);
  }
  if (count == 0 || plans[0]->n == 0) return GAR_OK;
  for (const gar_plan *pl : ps)
    if (int rc = check_fused_size(pl)) return rc;
  if (reinterpret_cast<uintptr_t>(desc) % 8 != 0) {
    set_error("descriptor array is not 8-byte aligned");
    return GAR_EALIGN;
  }
  CodegenResult cg = generate_batched_source(ps);
  JitKernel *k = nullptr;
  int rc = jit_compile(cg, &k);
  if (rc) return rc;
  rc = jit_load(k);
  if (rc) return rc;
  struct {
    const gar_batch_desc *desc;
    unsigned long long count;
  } a = {desc, (unsigned long long)count};
  void *kargs[] = {&a};
  const uint64_t per = plans[0]->n / k->width + plans[0]->n % k->width;
  const int grid = grid_for(k, per * (uint64_t)count);
  cudaError_t e = launch_generated(k, grid, kargs, stream);
  if (e != cudaSuccess) return cuda_fail(e, "batched kernel launch");
  return GAR_OK;
}

int gar_last_step_bytes(const gar_plan *pl, uint64_t *per_step) {
  if (int rc = check_plan(pl)) return rc;
  if (per_step == nullptr) return GAR_EINVAL;
  if (!pl->ran_step_faithful) {
    set_error("no step-faithful Allreduce has run on this plan");
    return GAR_ESTATE;
  }
  cudaError_t e = cudaStreamSynchronize((cudaStream_t)pl->last_stream);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  std::vector<unsigned long long> tmp((size_t)pl->S * STEP_BYTE_SLOTS);
  e = cudaMemcpy(tmp.data(), pl->d_step_bytes, tmp.size() * sizeof(unsigned long long),
                 cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy(step counters)");
  for (int t = 0; t < pl->S; ++t) {
    uint64_t sum = 0;
    for (int k = 0; k < STEP_BYTE_SLOTS; ++k) sum += tmp[(size_t)t * STEP_BYTE_SLOTS + k];
    per_step[t] = sum;
  }
  return GAR_OK;
}

int gar_plan_status(gar_plan *pl) {
  if (int rc = check_plan(pl)) return rc;
  if (!pl->ran_persistent || pl->d_barrier == nullptr) return GAR_OK;
  cudaError_t e = cudaStreamSynchronize((cudaStream_t)pl->last_stream);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  int st[4] = {0, 0, 0, 0};
  e = cudaMemcpy(st, pl->d_barrier, sizeof st, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy(barrier state)");
  if (st[2] != 0) {
    set_error("persistent step-faithful kernel: a grid-barrier wait gave up after launch " +
              std::to_string(st[3]));
    return GAR_ETIMEOUT;
  }
  return GAR_OK;
}

int gar_plan_debug_barrier(gar_plan *pl, unsigned int phantom, unsigned int spin_limit) {
  if (int rc = check_plan(pl)) return rc;
  pl->barrier_phantom = phantom;
  pl->barrier_spin_limit = spin_limit ? spin_limit : default_spin_limit(*pl);
  return GAR_OK;
}

const char *gar_strerror(int status) {
  switch (status) {
    case GAR_OK: return "success";
    case GAR_EINVAL: return "invalid argument";
    case GAR_ENOMEM: return "out of memory";
    case GAR_EALIGN: return "buffer not 16-byte aligned";
    case GAR_ECUDA: return "CUDA error";
    case GAR_EJIT: return "kernel compilation failed";
    case GAR_ENOWS: return "workspace missing or too small";
    case GAR_ESTATE: return "invalid plan state";
    case GAR_ETIMEOUT: return "bounded wait timed out";
  }
  return "unknown status";
}

const char *gar_last_error(void) { return last_error_cstr(); }

int gar_cost_model(int P, int steps, double m_bytes, double alpha, double beta, double gamma,
                   double *tau) {
  if (P < 1 || tau == nullptr) {
    set_error("bad cost-model arguments");
    return GAR_EINVAL;
  }
  const int L = ceil_log2(P);
  const double u = m_bytes / P;
  if (steps == GAR_STEPS_BO) steps = 2 * L;
  if (steps == GAR_STEPS_LO) steps = L;
  if (steps == GAR_STEPS_RING) {  // eq. naive_cost
    *tau = 2.0 * (P - 1) * alpha + 2.0 * (P - 1) * u * beta + (P - 1) * u * gamma;
    return GAR_OK;
  }
  if (steps > 2 * L && steps <= 2 * (P - 1) && steps % 2 == 0) {
    // fold schedule: the bandwidth-optimal traffic and combines in S steps (equals
    // eq. bo_cost at S = 2L and eq. naive_cost at S = 2(P-1))
    *tau = steps * alpha + 2.0 * (P - 1) * u * beta + (P - 1) * u * gamma;
    return GAR_OK;
  }
  const int r = 2 * L - steps;
  if (r < 0 || r > L) {
    set_error("steps outside [L, 2L], an even count up to 2(P-1), or GAR_STEPS_*");
    return GAR_EINVAL;
  }
  if (r == L) {  // latency-optimal, eq. lo_cost
    *tau = L * alpha + (double)P * L * u * beta + (double)P * (2.0 * L - 2.0) * u * gamma;
  } else {       // eq. intemediate_cost (r = 0 gives eq. bo_cost)
    const double extra = std::ldexp(1.0, r) - 1.0;
    *tau = (2.0 * L - r) * alpha + (2.0 * (P - 1) + extra * (L - 1)) * u * beta +
           ((P - 1) + extra * (2.0 * L - 2.0)) * u * gamma;
  }
  return GAR_OK;
}

int gar_optimal_steps(int P, double m_bytes, double alpha, double beta, double gamma, int *steps) {
  if (P < 1 || steps == nullptr) {
    set_error("bad cost-model arguments");
    return GAR_EINVAL;
  }
  const int L = ceil_log2(P);
  int best = L;
  double best_t = 0;
  for (int S = L; S <= 2 * L; ++S) {
    double t = 0;
    gar_cost_model(P, S, m_bytes, alpha, beta, gamma, &t);
    if (S == L || t < best_t - 1e-18) {
      best = S;
      best_t = t;
    }
  }
  *steps = best;
  return GAR_OK;
}

int gar_selftest_compile(void) {
  const int cases[][4] = {{24, GAR_F32, GAR_SUM, -1}, {7, GAR_F32, GAR_MAX, 3},
                          {5, GAR_BF16, GAR_SUM, 4},  {6, GAR_I32, GAR_MIN, 3}};
  for (const auto &c : cases) {
    gar_plan *pl = nullptr;
    int rc = gar_plan_create(&pl, c[0], 1000 + c[0], c[1], c[2], c[3]);
    if (rc) return rc;
    rc = gar_plan_compile(pl, GAR_FUSED);
    if (rc == GAR_OK) {
      std::vector<const gar_plan *> ps{pl};
      JitKernel *k = nullptr;
      rc = jit_compile(generate_batched_source(ps), &k);
    }
    gar_plan_destroy(pl);
    if (rc) return rc;
  }
  return GAR_OK;
}

}  // extern "C"
