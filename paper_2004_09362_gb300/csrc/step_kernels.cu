// Step-faithful mode: one kernel launch per communication step of the schedule.
//
// A launch applies the step's block ops (plan.cpp) for every rank x at once.  An op
// names a placement; rank x works on block b = (x - dst_place) mod P, which is the same
// block index at the partner (a move by t^{l} changes a vector's placement, never its
// block index; eq. comm_op_0).  "Sending" is a coalesced 16-byte vector read of the
// partner rank's block; the read value is combined in registers with the own block
// (eq. distr_vectors_combination) and stored.  Every CTA owns one chunk of one block
// of one (op, rank) pair (short blocks: one thread per (op, element) instead).  Combine
// ops batch 2 vectors per thread; same-type copies move raw 16-byte units, 6 per
// thread; a bf16 plan's first step keeps its 16-byte bf16 loads packed until the
// combine.  Each warp counts the elements it read from partners and adds the bytes to
// one of the step's counter slots, so the bytes a step actually moved are recorded.
// The launches of one Allreduce are chained by programmatic dependent launch.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <string>
#include <type_traits>

#include "gar_internal.hpp"

namespace gar {
namespace {

#ifndef GAR_STEP_CHUNK
#define GAR_STEP_CHUNK 16384
#endif
#ifndef GAR_STEP_UNROLL
#define GAR_STEP_UNROLL 2
#endif
// Launch shape, from a sweep on GB300 (P=24 x 64 MiB fp32, P=127 x 8 MiB bf16, P=8 x
// 1 MiB): CTAs own 16384-element chunks (smaller chunks ran up to 2.5x slower) and each
// thread issues the loads of 2 vectors before combining.  Small vectors drop the chunk
// to 8192 or 4096 elements to keep at least 4 CTAs per SM.
constexpr int kThreads = 256;
constexpr uint64_t kChunk = GAR_STEP_CHUNK;  // largest chunk (elements per CTA)
constexpr int kUnroll = GAR_STEP_UNROLL;     // 4-element vectors a thread loads at once
constexpr uint64_t kFlatBelow = 4 * kThreads * kUnroll;  // blocks shorter than this: element-major

template <int MAXP>
struct StepArgs {
  void *rank[MAXP];
  void *ws[NUM_WS_BUFS];             // QP0, QP1, QS slice bases (nullptr if unused)
  const StepOp *ops;                 // this launch's ops
  unsigned long long *bytes;         // STEP_BYTE_SLOTS counters of the step, or nullptr
  uint64_t q, rem, n_pad;
  uint64_t chunk;                    // elements per CTA
  uint64_t n;                        // elements per rank
  int P, partner, nops, nchunks;
  int xor_group;                     // 1: placements and partners combine by XOR (Table 1b)
};

template <typename T> struct AccOf { using type = T; };
template <> struct AccOf<__nv_bfloat16> { using type = float; };

__device__ __forceinline__ float widen(__nv_bfloat16 x) { return __bfloat162float(x); }
__device__ __forceinline__ float widen(float x) { return x; }
__device__ __forceinline__ int widen(int x) { return x; }
__device__ __forceinline__ void narrow(float x, __nv_bfloat16 *o) { *o = __float2bfloat16_rn(x); }
__device__ __forceinline__ void narrow(float x, float *o) { *o = x; }
__device__ __forceinline__ void narrow(int x, int *o) { *o = x; }

template <int OP> __device__ __forceinline__ float combine(float a, float b) {
  if (OP == GAR_SUM) return a + b;
  if (OP == GAR_MAX) return fmaxf(a, b);
  return fminf(a, b);
}
template <int OP> __device__ __forceinline__ int combine(int a, int b) {
  if (OP == GAR_SUM) return (int)((unsigned)a + (unsigned)b);
  if (OP == GAR_MAX) return a > b ? a : b;
  return a < b ? a : b;
}

// One element / four aligned elements of buffer `buf` (rank buffers hold T, workspace
// slices hold the accumulation type A).
template <typename T, typename A>
__device__ __forceinline__ A load1(uint8_t buf, const void *base, uint64_t e) {
  if (buf == BUF_RANK) return widen(static_cast<const T *>(base)[e]);
  return static_cast<const A *>(base)[e];
}

template <typename T, typename A>
__device__ __forceinline__ void load4(uint8_t buf, const void *base, uint64_t e, A (&v)[4]) {
  if (buf == BUF_RANK && sizeof(T) == 2) {
    const uint2 u = *reinterpret_cast<const uint2 *>(static_cast<const T *>(base) + e);
    v[0] = (A)__uint_as_float(u.x << 16);
    v[1] = (A)__uint_as_float(u.x & 0xffff0000u);
    v[2] = (A)__uint_as_float(u.y << 16);
    v[3] = (A)__uint_as_float(u.y & 0xffff0000u);
  } else {
    const A *p = (buf == BUF_RANK) ? reinterpret_cast<const A *>(static_cast<const T *>(base))
                                   : static_cast<const A *>(base);
    const int4 u = *reinterpret_cast<const int4 *>(p + e);
    v[0] = *reinterpret_cast<const A *>(&u.x);
    v[1] = *reinterpret_cast<const A *>(&u.y);
    v[2] = *reinterpret_cast<const A *>(&u.z);
    v[3] = *reinterpret_cast<const A *>(&u.w);
  }
}

template <typename T, typename A>
__device__ __forceinline__ void store1(uint8_t buf, void *base, uint64_t e, A v) {
  if (buf == BUF_RANK)
    narrow(v, static_cast<T *>(base) + e);
  else
    static_cast<A *>(base)[e] = v;
}

template <typename T, typename A>
__device__ __forceinline__ void store4(uint8_t buf, void *base, uint64_t e, const A (&v)[4]) {
  if (buf == BUF_RANK && sizeof(T) == 2) {
    __nv_bfloat16 h[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) narrow(v[k], &h[k]);
    uint2 u;
    u.x = (uint32_t)__bfloat16_as_ushort(h[0]) | ((uint32_t)__bfloat16_as_ushort(h[1]) << 16);
    u.y = (uint32_t)__bfloat16_as_ushort(h[2]) | ((uint32_t)__bfloat16_as_ushort(h[3]) << 16);
    *reinterpret_cast<uint2 *>(static_cast<T *>(base) + e) = u;
  } else {
    A *p = (buf == BUF_RANK) ? reinterpret_cast<A *>(static_cast<T *>(base)) : static_cast<A *>(base);
    int4 u;
    u.x = *reinterpret_cast<const int *>(&v[0]);
    u.y = *reinterpret_cast<const int *>(&v[1]);
    u.z = *reinterpret_cast<const int *>(&v[2]);
    u.w = *reinterpret_cast<const int *>(&v[3]);
    *reinterpret_cast<int4 *>(p + e) = u;
  }
}

template <typename A, int MAXP>
__device__ __forceinline__ void *buf_ptr(const StepArgs<MAXP> &a, uint8_t buf, int rank) {
  if (buf == BUF_RANK) return a.rank[rank];
  if (buf == BUF_NONE) return nullptr;
  return static_cast<char *>(a.ws[buf - BUF_QP0]) + (uint64_t)rank * a.n_pad * sizeof(A);
}

// v mod P for v in (-P, 2P).
__device__ __forceinline__ int wrap_rank(int v, int P) { return v < 0 ? v + P : (v >= P ? v - P : v); }

// This warp's slot of a step's byte counter.
__device__ __forceinline__ int byte_slot() {
  return (int)((blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5)) % STEP_BYTE_SLOTS);
}

// Per-launch parameters the work functions need besides the buffers.
struct LaunchView {
  const StepOp *ops;
  unsigned long long *bytes;  // STEP_BYTE_SLOTS counters of the communication step, or nullptr
  uint64_t chunk;             // elements per CTA item (chunked mapping)
  int nops, partner, nchunks;
};

// Chunked mapping: work item `item` = (chunk, rank x, op) is done by the whole CTA.
// kCopyPaths: copy-only ops take the deeper copy loops.  The persistent kernel, which
// keeps its launch loop's state live around this body, leaves them out: with them it
// needs 109 registers (2 CTAs per SM) instead of about 75 (3 CTAs per SM).
template <typename T, int OP, int MAXP, bool kCopyPaths = true>
__device__ __forceinline__ void chunk_work(const StepArgs<MAXP> &a, const LaunchView &lv, uint64_t item) {
  using A = typename AccOf<T>::type;
  // 32-bit index arithmetic whenever the item fits (always for a launch's own grid):
  // 64-bit division is a long software sequence and ran once per CTA.
  int chunk, x, oi;
  if (item <= 0xffffffffull) {
    uint32_t it = (uint32_t)item;
    chunk = (int)(it % (uint32_t)lv.nchunks);
    it /= (uint32_t)lv.nchunks;
    x = (int)(it % (uint32_t)a.P);
    oi = (int)(it / (uint32_t)a.P);
  } else {
    chunk = (int)(item % (uint64_t)lv.nchunks);
    item /= (uint64_t)lv.nchunks;
    x = (int)(item % (uint64_t)a.P);
    oi = (int)(item / (uint64_t)a.P);
  }
  if (oi >= lv.nops) return;
  const StepOp op = lv.ops[oi];
  // placements and ranks are in [0, P), partner offsets in (-P, P)
  const int b = a.xor_group ? (x ^ (int)op.dst_place) : wrap_rank(x - (int)op.dst_place, a.P);
  const uint64_t bstart = (uint64_t)b * a.q + ((uint64_t)b < a.rem ? (uint64_t)b : a.rem);
  const uint64_t blen = a.q + ((uint64_t)b < a.rem ? 1 : 0);
  const uint64_t c0 = (uint64_t)chunk * lv.chunk;
  if (c0 >= blen) return;
  const uint64_t lo = bstart + c0;
  const uint64_t hi = bstart + (blen < c0 + lv.chunk ? blen : c0 + lv.chunk);

  const bool has_recv = op.recv_place >= 0;
  const int partner = a.xor_group ? (x ^ lv.partner) : wrap_rank(x + lv.partner, a.P);
  const void *recv = has_recv ? buf_ptr<A>(a, op.recv_buf, partner) : nullptr;
  void *out0 = buf_ptr<A>(a, op.out0_buf, x);
  const void *own0 = buf_ptr<A>(a, op.out0_own, x);
  void *out1 = buf_ptr<A>(a, op.out1_buf, x);
  const void *own1 = buf_ptr<A>(a, op.out1_own, x);

  uint64_t moved = 0;
  auto do1 = [&](uint64_t e) {
    A r = A(0);
    if (has_recv) {
      r = load1<T, A>(op.recv_buf, recv, e);
      ++moved;
    }
    A o0 = r, o1 = r;
    if (own0) o0 = has_recv ? combine<OP>(load1<T, A>(op.out0_own, own0, e), r) : load1<T, A>(op.out0_own, own0, e);
    if (out1 && own1) o1 = has_recv ? combine<OP>(load1<T, A>(op.out1_own, own1, e), r) : load1<T, A>(op.out1_own, own1, e);
    store1<T, A>(op.out0_buf, out0, e, o0);
    if (out1) store1<T, A>(op.out1_buf, out1, e, o1);
  };
  // kUnroll aligned 4-element vectors per thread: every load of the batch is issued
  // before the first combine, so a thread keeps up to 3 * kUnroll 16-byte loads in flight.
  auto do4xU = [&](uint64_t e_first, uint64_t stride, uint64_t vend) {
    A r[kUnroll][4], o0[kUnroll][4], o1[kUnroll][4];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const uint64_t e = e_first + u * stride;
      if (e < vend) {
        if (has_recv) {
          load4<T, A>(op.recv_buf, recv, e, r[u]);
          moved += 4;
        }
        if (own0) load4<T, A>(op.out0_own, own0, e, o0[u]);
        if (out1 && own1) load4<T, A>(op.out1_own, own1, e, o1[u]);
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const uint64_t e = e_first + u * stride;
      if (e < vend) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          if (!has_recv) {
            r[u][k] = A(0);
          }
          o0[u][k] = own0 ? (has_recv ? combine<OP>(o0[u][k], r[u][k]) : o0[u][k]) : r[u][k];
          if (out1) o1[u][k] = own1 ? (has_recv ? combine<OP>(o1[u][k], r[u][k]) : o1[u][k]) : r[u][k];
        }
        store4<T, A>(op.out0_buf, out0, e, o0[u]);
        if (out1) store4<T, A>(op.out1_buf, out1, e, o1[u]);
      }
    }
  };

  // Copy-only ops (one source, one output: the distribution steps' copies and the q*
  // moves) load one operand per vector instead of two, so they batch twice as many
  // vectors per thread to keep the same bytes in flight.
  auto copy4xU = [&](uint64_t e_first, uint64_t stride, uint64_t vend) {
    constexpr int U = 2 * kUnroll;
    const void *src = has_recv ? recv : own0;
    const uint8_t sbuf = has_recv ? op.recv_buf : op.out0_own;
    A v[U][4];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint64_t e = e_first + u * stride;
      if (e < vend) {
        load4<T, A>(sbuf, src, e, v[u]);
        if (has_recv) moved += 4;
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint64_t e = e_first + u * stride;
      if (e < vend) store4<T, A>(op.out0_buf, out0, e, v[u]);
    }
  };
  const bool copy_only = kCopyPaths && !out1 && (has_recv != (own0 != nullptr));
  const uint8_t copy_src_buf = has_recv ? op.recv_buf : op.out0_own;
  // A copy between buffers of one element type moves raw 16-byte units (4 fp32 or 8 bf16
  // elements) with a compile-time stride: few registers, so 6 units per thread in flight
  // within the 40-register budget.  bf16 copies used 8-byte units before and ran at
  // about 4 TB/s (48 bytes in flight per thread) against 6.6 TB/s for fp32; elements
  // before the first and after the last 16-byte boundary go one by one.
  auto raw_copy = [&](uint64_t va, uint64_t vb) {
    constexpr int U = 6;
    const void *srcp = has_recv ? recv : own0;
    const uint64_t esz = copy_src_buf == BUF_RANK ? sizeof(T) : sizeof(A);
    const uint64_t epu = 16 / esz;  // elements per 16-byte unit
    uint64_t ua = (va + epu - 1) / epu * epu, ub = vb / epu * epu;
    if (ua > vb) ua = vb;
    if (ub < ua) ub = ua;
    for (uint64_t e = va + threadIdx.x; e < ua; e += kThreads) do1(e);
    for (uint64_t e = ub + threadIdx.x; e < vb; e += kThreads) do1(e);
    const int4 *src = reinterpret_cast<const int4 *>(static_cast<const char *>(srcp) + ua * esz);
    int4 *dst = reinterpret_cast<int4 *>(static_cast<char *>(out0) + ua * esz);
    const uint64_t units = (ub - ua) / epu;
    for (uint64_t k = threadIdx.x; k < units; k += (uint64_t)U * kThreads) {
      const uint64_t left = units - k;
      int4 v[U];
#pragma unroll
      for (int u = 0; u < U; ++u)
        if ((uint64_t)u * kThreads < left) v[u] = src[k + (uint64_t)u * kThreads];
#pragma unroll
      for (int u = 0; u < U; ++u)
        if ((uint64_t)u * kThreads < left) dst[k + (uint64_t)u * kThreads] = v[u];
      if (has_recv) {
        const uint64_t cnt = left < (uint64_t)(U - 1) * kThreads + 1 ? (left + kThreads - 1) / kThreads : U;
        moved += epu * cnt;
      }
    }
  };
  const bool raw = copy_only && (sizeof(T) == sizeof(A) || copy_src_buf == op.out0_buf);

  // bf16 partner block + bf16 own block -> fp32 partial (the first reduction step of a
  // bf16 plan).  Each lane reads 4 bf16 (8 bytes) of both operands and writes their 4
  // fp32 partials as one 16-byte store, so every warp store covers 512 contiguous bytes.
  // Reading 8 bf16 per lane instead made each 16-byte store half of a 32-byte stretch, a
  // warp store then half-filled 32 sectors, and the step ran at 74 % of DRAM throughput
  // (P = 127 x 8 MiB bf16: whole Allreduce S = 14 1.190 -> 1.164 ms, S = 10 2.323 ->
  // 2.288 ms).  4 units per thread keep 64 bytes of loads in flight.
  auto packed_combine = [&](uint64_t va, uint64_t vb) {
    constexpr int U = 4;
    uint64_t ua = (va + 3) & ~uint64_t(3), ub = vb & ~uint64_t(3);
    if (ua > vb) ua = vb;
    if (ub < ua) ub = ua;
    for (uint64_t e = va + threadIdx.x; e < ua; e += kThreads) do1(e);
    for (uint64_t e = ub + threadIdx.x; e < vb; e += kThreads) do1(e);
    const uint2 *rp = reinterpret_cast<const uint2 *>(static_cast<const char *>(recv) + ua * sizeof(T));
    const uint2 *op_ = reinterpret_cast<const uint2 *>(static_cast<const char *>(own0) + ua * sizeof(T));
    float4 *dp = reinterpret_cast<float4 *>(static_cast<char *>(out0) + ua * sizeof(A));
    const uint64_t units = (ub - ua) >> 2;
    for (uint64_t k = threadIdx.x; k < units; k += (uint64_t)U * kThreads) {
      const uint64_t left = units - k;
      uint2 rv[U], ov[U];
#pragma unroll
      for (int u = 0; u < U; ++u)
        if ((uint64_t)u * kThreads < left) {
          rv[u] = rp[k + (uint64_t)u * kThreads];
          ov[u] = op_[k + (uint64_t)u * kThreads];
        }
#pragma unroll
      for (int u = 0; u < U; ++u)
        if ((uint64_t)u * kThreads < left) {
          float4 f;
          f.x = combine<OP>(__uint_as_float(ov[u].x << 16), __uint_as_float(rv[u].x << 16));
          f.y = combine<OP>(__uint_as_float(ov[u].x & 0xffff0000u), __uint_as_float(rv[u].x & 0xffff0000u));
          f.z = combine<OP>(__uint_as_float(ov[u].y << 16), __uint_as_float(rv[u].y << 16));
          f.w = combine<OP>(__uint_as_float(ov[u].y & 0xffff0000u), __uint_as_float(rv[u].y & 0xffff0000u));
          dp[k + (uint64_t)u * kThreads] = f;
        }
      if (has_recv) {
        const uint64_t cnt = left < (uint64_t)(U - 1) * kThreads + 1 ? (left + kThreads - 1) / kThreads : U;
        moved += cnt << 2;
      }
    }
  };
  const bool packed = sizeof(T) == 2 && kCopyPaths && has_recv && !out1 && own0 != nullptr &&
                      op.recv_buf == BUF_RANK && op.out0_own == BUF_RANK && op.out0_buf != BUF_RANK;

  // Element offsets are the same in every buffer, and every buffer base is 16-byte
  // aligned, so one head/body/tail split serves all operands.
  uint64_t va = (lo + 3) & ~uint64_t(3);
  uint64_t vb = hi & ~uint64_t(3);
  if (va > hi) va = hi;
  if (vb < va) vb = va;
  for (uint64_t e = lo + threadIdx.x; e < va; e += blockDim.x) do1(e);
  const uint64_t vstride = 4 * (uint64_t)blockDim.x;
  if (raw) {
    raw_copy(va, vb);
  } else if (packed) {
    packed_combine(va, vb);
  } else if (copy_only) {
    for (uint64_t e = va + 4 * (uint64_t)threadIdx.x; e < vb; e += 2 * kUnroll * vstride)
      copy4xU(e, vstride, vb);
  } else {
    for (uint64_t e = va + 4 * (uint64_t)threadIdx.x; e < vb; e += kUnroll * vstride)
      do4xU(e, vstride, vb);
  }
  for (uint64_t e = vb + threadIdx.x; e < hi; e += blockDim.x) do1(e);

  // The step's received bytes: summed over the warp, then over the CTA in shared memory,
  // one atomic add per CTA into one of the step's 32 counter slots.  (Whether an op
  // receives is the same for the whole CTA, so every thread takes this branch or none.)
  if (lv.bytes != nullptr && has_recv) {
    __shared__ unsigned long long s_moved[kThreads / 32];
    unsigned long long m = moved;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) m += __shfl_down_sync(0xffffffffu, m, off);
    if ((threadIdx.x & 31) == 0) s_moved[threadIdx.x >> 5] = m;
    __syncthreads();
    if (threadIdx.x == 0) {
      unsigned long long t = 0;
#pragma unroll
      for (int w = 0; w < kThreads / 32; ++w) t += s_moved[w];
      const unsigned long long esize = (op.recv_buf == BUF_RANK) ? sizeof(T) : sizeof(A);
      if (t) atomicAdd(lv.bytes + blockIdx.x % STEP_BYTE_SLOTS, t * esize);
    }
    __syncthreads();  // s_moved is written again by the next work item of a persistent CTA
  }
}

// Element-major mapping, for small blocks: an op touches block b = (x - dst_place) mod P
// at every rank x, i.e. every element position exactly once across the P ranks, so
// work item g = (op, element e) maps to rank x = (b(e) + dst_place) mod P.  One thread
// per item keeps every thread busy however short the blocks are.  Threads g_first,
// g_first + g_stride, ... of the launch's nops * n items.
template <typename T, int OP, int MAXP>
__device__ __forceinline__ void flat_work(const StepArgs<MAXP> &a, const LaunchView &lv, uint64_t g_first,
                                          uint64_t g_stride) {
  using A = typename AccOf<T>::type;
  const uint64_t total = (uint64_t)lv.nops * a.n;
  const uint64_t big = a.rem * (a.q + 1);
  unsigned long long moved_bytes = 0;
  // 32-bit index arithmetic when every index fits (the element-major launch serves
  // short blocks, so practically always): 64-bit division is a long software sequence.
  const bool narrow_idx = total + g_stride <= 0xffffffffull;
  for (uint64_t g = g_first; g < total; g += g_stride) {
    int oi, b;
    uint64_t e;
    if (narrow_idx) {
      const uint32_t g32 = (uint32_t)g, n32 = (uint32_t)a.n;
      oi = (int)(g32 / n32);
      const uint32_t e32 = g32 - (uint32_t)oi * n32;
      e = e32;
      b = e32 < (uint32_t)big ? (int)(e32 / (uint32_t)(a.q + 1))
                              : (int)((uint32_t)a.rem + (e32 - (uint32_t)big) / (uint32_t)a.q);
    } else {
      oi = (int)(g / a.n);
      e = g - (uint64_t)oi * a.n;
      b = e < big ? (int)(e / (a.q + 1)) : (int)(a.rem + (e - big) / a.q);
    }
    const StepOp op = lv.ops[oi];
    const int x = a.xor_group ? (b ^ (int)op.dst_place) : wrap_rank(b + (int)op.dst_place, a.P);
    A r = A(0);
    const bool has_recv = op.recv_place >= 0;
    if (has_recv) {
      const int partner = a.xor_group ? (x ^ lv.partner) : wrap_rank(x + lv.partner, a.P);
      r = load1<T, A>(op.recv_buf, buf_ptr<A>(a, op.recv_buf, partner), e);
      moved_bytes += (op.recv_buf == BUF_RANK) ? sizeof(T) : sizeof(A);
    }
    A o0 = r, o1 = r;
    if (op.out0_own != BUF_NONE) {
      const A v = load1<T, A>(op.out0_own, buf_ptr<A>(a, op.out0_own, x), e);
      o0 = has_recv ? combine<OP>(v, r) : v;
    }
    if (op.out1_buf != BUF_NONE && op.out1_own != BUF_NONE) {
      const A v = load1<T, A>(op.out1_own, buf_ptr<A>(a, op.out1_own, x), e);
      o1 = has_recv ? combine<OP>(v, r) : v;
    }
    store1<T, A>(op.out0_buf, buf_ptr<A>(a, op.out0_buf, x), e, o0);
    if (op.out1_buf != BUF_NONE) store1<T, A>(op.out1_buf, buf_ptr<A>(a, op.out1_buf, x), e, o1);
  }
  if (lv.bytes != nullptr) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) moved_bytes += __shfl_down_sync(0xffffffffu, moved_bytes, off);
    if ((threadIdx.x & 31) == 0 && moved_bytes) atomicAdd(lv.bytes + byte_slot(), moved_bytes);
  }
}

template <int MAXP>
__device__ __forceinline__ LaunchView view_of(const StepArgs<MAXP> &a) {
  LaunchView lv;
  lv.ops = a.ops;
  lv.bytes = a.bytes;
  lv.chunk = a.chunk;
  lv.nops = a.nops;
  lv.partner = a.partner;
  lv.nchunks = a.nchunks;
  return lv;
}

// Programmatic dependent launch: the step launches of one Allreduce are made with
// programmatic stream serialisation, so launch i+1's CTAs may become resident while
// launch i drains.  griddepcontrol.wait blocks until every prerequisite grid has
// completed and its memory is visible (a no-op without such a dependency); nothing is
// read before it.  launch_dependents, issued once a CTA's work is done, lets the next
// launch start once every CTA of this one has issued it or exited.
__device__ __forceinline__ void wait_prior_grid() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void allow_next_grid() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// At most 40 registers (6 CTAs per SM): the bf16 launches ran 5-8 % faster than at the
// 48 registers the compiler picks unbounded, fp32 the same.
template <typename T, int OP, int MAXP>
__global__ void __launch_bounds__(kThreads, 6) step_kernel(const __grid_constant__ StepArgs<MAXP> a) {
  wait_prior_grid();
  chunk_work<T, OP, MAXP>(a, view_of(a), blockIdx.x);
  allow_next_grid();
}

template <typename T, int OP, int MAXP>
__global__ void __launch_bounds__(kThreads) step_kernel_flat(const __grid_constant__ StepArgs<MAXP> a) {
  wait_prior_grid();
  flat_work<T, OP, MAXP>(a, view_of(a), (uint64_t)blockIdx.x * blockDim.x + threadIdx.x,
                         (uint64_t)gridDim.x * blockDim.x);
  allow_next_grid();
}

// Launches a step kernel with programmatic stream serialisation (see above).
template <typename Args>
cudaError_t launch_pdl(void (*kernel)(Args), unsigned grid, gar_stream_t stream, const Args &a) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = (cudaStream_t)stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, a);
}

// ---------------------------------------------------------------------------
// Persistent step-faithful mode (GAR_STEP_PERSISTENT): one cooperative launch runs every
// step of the schedule; a grid-wide barrier between steps takes the place of the kernel
// boundary.  The barrier's waits are bounded: after spin_limit polls a CTA records a
// timeout in the barrier state and returns, and every other CTA stops at its next poll,
// so the kernel always ends and the context stays usable; the host reads the outcome
// with gar_plan_status.
// ---------------------------------------------------------------------------

struct BarrierState {
  unsigned int count;   // CTA arrivals since the launch began (zeroed before each launch)
  unsigned int unused;
  int error;            // 1 once any CTA gave up waiting
  int error_launch;     // launch index after which the first timeout happened
};

template <int MAXP>
struct PersistArgs {
  StepArgs<MAXP> s;                 // buffers and sizes (s.ops = whole op table)
  const LaunchDesc *launches;
  unsigned long long *step_bytes;   // per communication step, or nullptr
  BarrierState *bar;
  int nlaunch;
  int flat;                         // element-major mapping (small blocks)
  unsigned int spin_limit;          // polls before a wait gives up
  unsigned int phantom;             // arrivals expected beyond the grid (test hook, normally 0)
};

__device__ __forceinline__ unsigned ld_acquire_gpu(const unsigned *p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ unsigned atom_add_acq_rel_gpu(unsigned *p, unsigned v) {
  unsigned old;
  asm volatile("atom.add.acq_rel.gpu.global.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}
__device__ __forceinline__ int ld_relaxed_int(const int *p) {
  int v;
  asm volatile("ld.relaxed.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Grid-wide barrier number `launch` (0-based) with a bounded wait.  Every CTA adds one
// to the arrival count with acquire-release semantics (release: the CTA's writes of the
// step, ordered before it by __syncthreads, become visible with it; acquire: the CTA
// that arrives last reads the others' writes, having seen all their arrivals in the add
// itself) and polls the count with acquire loads until it reaches (launch + 1) *
// expected, the arrivals of this and every earlier barrier of the launch.  The count
// only grows within a launch, so no CTA resets it and the last arrival releases everyone
// at once.  Returns false (for the whole CTA) if this or any other CTA timed out.
__device__ bool grid_barrier(BarrierState *bar, unsigned expected, unsigned spin_limit, int launch) {
  __shared__ int s_ok;
  __syncthreads();
  if (threadIdx.x == 0) {
    int ok = 1;
    const unsigned target = (unsigned)(launch + 1) * expected;
    unsigned now = atom_add_acq_rel_gpu(&bar->count, 1u) + 1u;
    unsigned polls = 0;
    while (now < target) {
      ++polls;
      if (polls >= spin_limit || ((polls & 63u) == 0 && ld_relaxed_int(&bar->error) != 0)) {
        ok = 0;
        break;
      }
      if (polls > 32) __nanosleep(32);
      now = ld_acquire_gpu(&bar->count);
    }
    if (!ok && atomicCAS(&bar->error, 0, 1) == 0) bar->error_launch = launch;
    s_ok = ok;
  }
  __syncthreads();
  return s_ok != 0;
}

template <typename T, int OP, int MAXP>
__global__ void __launch_bounds__(kThreads) step_kernel_persistent(const __grid_constant__ PersistArgs<MAXP> p) {
  const unsigned expected = gridDim.x + p.phantom;
  for (int l = 0; l < p.nlaunch; ++l) {
    const LaunchDesc d = p.launches[l];
    LaunchView lv;
    lv.ops = p.s.ops + d.first_op;
    lv.nops = d.nops;
    lv.partner = d.partner;
    lv.bytes = (p.step_bytes != nullptr && d.comm_step >= 0)
                   ? p.step_bytes + (size_t)d.comm_step * STEP_BYTE_SLOTS : nullptr;
    lv.chunk = p.s.chunk;
    lv.nchunks = p.s.nchunks;
    if (p.flat) {
      flat_work<T, OP, MAXP>(p.s, lv, (uint64_t)blockIdx.x * blockDim.x + threadIdx.x,
                             (uint64_t)gridDim.x * blockDim.x);
    } else {
      const uint64_t items = (uint64_t)lv.nchunks * (uint64_t)p.s.P * (uint64_t)lv.nops;
      for (uint64_t item = blockIdx.x; item < items; item += gridDim.x)
        chunk_work<T, OP, MAXP, false>(p.s, lv, item);
    }
    if (l + 1 < p.nlaunch && !grid_barrier(p.bar, expected, p.spin_limit, l)) return;
  }
}

// SM count of the current device (cached per device ordinal).
int num_sms() {
  static int cache[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) {
    cudaGetLastError();
    dev = 0;
  }
  if (dev < 64 && cache[dev] > 0) return cache[dev];
  int v = 0;
  if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0) {
    cudaGetLastError();
    v = 1;
  }
  if (dev < 64) cache[dev] = v;
  return v;
}

template <typename T, int OP, int MAXP>
int launch_typed(const gar_plan &pl, const Launch &ln, int launch_index, void *const *rank,
                 gar_stream_t stream) {
  (void)launch_index;
  StepArgs<MAXP> a{};
  for (int x = 0; x < pl.P; ++x) a.rank[x] = rank[x];
  int slot = 0;
  for (int k = 0; k < NUM_WS_BUFS; ++k) {
    if (pl.ws_used[k]) {
      a.ws[k] = static_cast<char *>(pl.ws) + (size_t)slot * pl.P * pl.n_pad * acc_size(pl.dtype);
      ++slot;
    } else {
      a.ws[k] = nullptr;
    }
  }
  a.ops = pl.d_ops + ln.first_op;
  a.bytes = (ln.comm_step >= 0) ? pl.d_step_bytes + (size_t)ln.comm_step * STEP_BYTE_SLOTS : nullptr;
  a.q = pl.q;
  a.rem = pl.rem;
  a.n_pad = pl.n_pad;
  a.n = pl.n;
  a.P = pl.P;
  a.xor_group = pl.group == GAR_GROUP_XOR ? 1 : 0;
  a.partner = ln.partner;
  a.nops = ln.nops;
  const uint64_t maxblk = pl.q + (pl.rem ? 1 : 0);
  if (maxblk < kFlatBelow && ln.nops > 0 && pl.n > 0) {
    // blocks shorter than one CTA's worth of vectors: element-major launch
    const uint64_t total = (uint64_t)ln.nops * pl.n;
    const uint64_t grid = std::min<uint64_t>((total + kThreads - 1) / kThreads,
                                             (uint64_t)num_sms() * 32);
    cudaError_t e = launch_pdl(step_kernel_flat<T, OP, MAXP>, (unsigned)grid, stream, a);
    if (e != cudaSuccess) return cuda_fail(e, "step kernel launch");
    return GAR_OK;
  }
  // Distribution steps copy 2-byte elements with as many bytes per CTA as fp32 chunks
  // hold; a last chunk shorter than 1/8 of a chunk is spread over the block's others (P =
  // 127 x 8 MiB bf16: blocks of 33,026 elements became 16,384 + 16,384 + 258, a third of
  // the CTAs nearly empty).
  a.chunk = (ln.phase == 1 && sizeof(T) == 2) ? 2 * kChunk : kChunk;
  const uint64_t min_ctas = 4 * (uint64_t)num_sms();
  while (a.chunk > 4096 && ((maxblk + a.chunk - 1) / a.chunk) * pl.P * ln.nops < min_ctas) a.chunk /= 2;
  {
    const uint64_t nch = (maxblk + a.chunk - 1) / a.chunk;
    if (nch > 1 && maxblk - (nch - 1) * a.chunk < a.chunk / 8)
      a.chunk = ((maxblk + nch - 2) / (nch - 1) + 7) / 8 * 8;
  }
  a.nchunks = (int)((maxblk + a.chunk - 1) / a.chunk);
  if (a.nchunks == 0 || ln.nops == 0) return GAR_OK;
  const uint64_t grid = (uint64_t)a.nchunks * (uint64_t)pl.P * (uint64_t)ln.nops;
  if (grid > 0x7fffffffull) {
    set_error("step launch grid too large");
    return GAR_EINVAL;
  }
  cudaError_t e = launch_pdl(step_kernel<T, OP, MAXP>, (unsigned)grid, stream, a);
  if (e != cudaSuccess) return cuda_fail(e, "step kernel launch");
  return GAR_OK;
}

template <typename T, int MAXP>
int launch_op(const gar_plan &pl, const Launch &ln, int li, void *const *rank, gar_stream_t s) {
  switch (pl.op) {
    case GAR_SUM: return launch_typed<T, GAR_SUM, MAXP>(pl, ln, li, rank, s);
    case GAR_MAX: return launch_typed<T, GAR_MAX, MAXP>(pl, ln, li, rank, s);
    case GAR_MIN: return launch_typed<T, GAR_MIN, MAXP>(pl, ln, li, rank, s);
  }
  return GAR_EINVAL;
}

template <int MAXP>
int launch_dt(const gar_plan &pl, const Launch &ln, int li, void *const *rank, gar_stream_t s) {
  switch (pl.dtype) {
    case GAR_F32: return launch_op<float, MAXP>(pl, ln, li, rank, s);
    case GAR_BF16: return launch_op<__nv_bfloat16, MAXP>(pl, ln, li, rank, s);
    case GAR_I32: return launch_op<int, MAXP>(pl, ln, li, rank, s);
  }
  return GAR_EINVAL;
}

template <typename T, int OP, int MAXP>
int launch_persistent_typed(const gar_plan &pl, void *const *rank, gar_stream_t stream) {
  PersistArgs<MAXP> p{};
  for (int x = 0; x < pl.P; ++x) p.s.rank[x] = rank[x];
  int slot = 0;
  for (int k = 0; k < NUM_WS_BUFS; ++k)
    p.s.ws[k] = pl.ws_used[k] ? static_cast<char *>(pl.ws) + (size_t)(slot++) * pl.P * pl.n_pad * acc_size(pl.dtype)
                              : nullptr;
  p.s.ops = pl.d_ops;
  p.s.bytes = nullptr;
  p.s.q = pl.q;
  p.s.rem = pl.rem;
  p.s.n_pad = pl.n_pad;
  p.s.n = pl.n;
  p.s.P = pl.P;
  p.s.xor_group = pl.group == GAR_GROUP_XOR ? 1 : 0;
  const uint64_t maxblk = pl.q + (pl.rem ? 1 : 0);
  p.flat = maxblk < kFlatBelow ? 1 : 0;
  // chunks as the per-step launches choose them for their largest step: small vectors
  // drop to 8192 or 4096 elements so that the grid has work for every CTA it can hold
  int max_ops = 1;
  for (const Launch &ln : pl.launches) max_ops = std::max(max_ops, ln.nops);
  p.s.chunk = kChunk;
  const uint64_t min_items = 4 * (uint64_t)num_sms();
  while (p.s.chunk > 4096 && ((maxblk + p.s.chunk - 1) / p.s.chunk) * pl.P * max_ops < min_items) p.s.chunk /= 2;
  p.s.nchunks = (int)((maxblk + p.s.chunk - 1) / p.s.chunk);
  p.launches = static_cast<const LaunchDesc *>(pl.d_launches);
  p.step_bytes = pl.d_step_bytes;
  p.bar = static_cast<BarrierState *>(pl.d_barrier);
  p.nlaunch = (int)pl.launches.size();
  p.spin_limit = pl.barrier_spin_limit;
  p.phantom = pl.barrier_phantom;
  const void *fn = (const void *)step_kernel_persistent<T, OP, MAXP>;
  int per_sm = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kThreads, 0);
  if (e != cudaSuccess || per_sm < 1) return cuda_fail(e == cudaSuccess ? cudaErrorInvalidConfiguration : e,
                                                       "persistent kernel occupancy");
  // As many CTAs as the largest step has work items (one chunk of one block op, or 256
  // element-major items), at most the co-resident maximum: a small Allreduce then waits
  // at its barriers for a few CTAs instead of three per SM.
  uint64_t need = 1;
  for (const Launch &ln : pl.launches) {
    const uint64_t items = p.flat ? ((uint64_t)ln.nops * pl.n + kThreads - 1) / kThreads
                                  : (uint64_t)p.s.nchunks * (uint64_t)pl.P * (uint64_t)ln.nops;
    need = std::max(need, items);
  }
  const unsigned grid = (unsigned)std::min<uint64_t>(need, (uint64_t)per_sm * (uint64_t)num_sms());
  void *args[] = {&p};
  e = cudaLaunchCooperativeKernel(fn, dim3(grid), dim3(kThreads), args, 0, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "persistent kernel launch");
  return GAR_OK;
}

template <typename T, int MAXP>
int launch_persistent_op(const gar_plan &pl, void *const *rank, gar_stream_t s) {
  switch (pl.op) {
    case GAR_SUM: return launch_persistent_typed<T, GAR_SUM, MAXP>(pl, rank, s);
    case GAR_MAX: return launch_persistent_typed<T, GAR_MAX, MAXP>(pl, rank, s);
    case GAR_MIN: return launch_persistent_typed<T, GAR_MIN, MAXP>(pl, rank, s);
  }
  return GAR_EINVAL;
}

template <int MAXP>
int launch_persistent_dt(const gar_plan &pl, void *const *rank, gar_stream_t s) {
  switch (pl.dtype) {
    case GAR_F32: return launch_persistent_op<float, MAXP>(pl, rank, s);
    case GAR_BF16: return launch_persistent_op<__nv_bfloat16, MAXP>(pl, rank, s);
    case GAR_I32: return launch_persistent_op<int, MAXP>(pl, rank, s);
  }
  return GAR_EINVAL;
}

}  // namespace

int launch_step(const gar_plan &pl, const Launch &ln, int launch_index, void *const *rank,
                gar_stream_t stream) {
  if (pl.P <= 128) return launch_dt<128>(pl, ln, launch_index, rank, stream);
  return launch_dt<GAR_MAX_P>(pl, ln, launch_index, rank, stream);
}

int launch_persistent(const gar_plan &pl, void *const *rank, gar_stream_t stream) {
  if (pl.P <= 128) return launch_persistent_dt<128>(pl, rank, stream);
  return launch_persistent_dt<GAR_MAX_P>(pl, rank, stream);
}

size_t barrier_state_bytes() { return sizeof(BarrierState); }

}  // namespace gar

// ---------------------------------------------------------------------------
// Step-faithful Allreduce without device allocation (gar_allreduce_noalloc).
//
// For callers that must not allocate device memory at call time -- code running
// under a caching allocator that owns all of the GPU's memory, or a host runtime with
// no allocator hook -- the workspace lives in one file-scope device array of fixed
// size instead of a caller-supplied buffer, and each launch receives its block ops by
// value in the kernel parameters instead of from a device table.  No cudaMalloc,
// cudaFree or memset is issued.  The array exists on a device once this file's device
// code is loaded there -- under CUDA's lazy module loading, at the first launch of any
// of its kernels, at gar_plan_prepare of a step-faithful mode, or at the first
// no-allocation call -- and stays until the process exits.  Nothing in it needs to
// start at zero: the schedule writes every workspace slot before it reads it.  All
// calls share the array, so two calls whose work overlaps on the GPU race.
// ---------------------------------------------------------------------------

static __device__ __align__(256) unsigned char g_noalloc_scratch[GAR_NOALLOC_SCRATCH_BYTES];

namespace gar {
namespace {

constexpr int kNoAllocMaxOps = 2 * GAR_NOALLOC_MAX_P;  // |transmit set| + K <= 2P per launch

struct NoAllocArgs {
  void *rank[GAR_NOALLOC_MAX_P];
  void *ws[NUM_WS_BUFS];
  StepOp ops[kNoAllocMaxOps];
  uint64_t q, rem, n_pad;
  int P, partner, nops, nchunks;
};

template <typename A>
__device__ __forceinline__ void *na_buf_ptr(const NoAllocArgs &a, uint8_t buf, int rank) {
  if (buf == BUF_RANK) return a.rank[rank];
  if (buf == BUF_NONE) return nullptr;
  return static_cast<char *>(a.ws[buf - BUF_QP0]) + (uint64_t)rank * a.n_pad * sizeof(A);
}

// Same block-op semantics as step_kernel (one CTA per op x rank x chunk), with the ops
// read from the parameter block and no byte counting.
template <typename T, int OP>
__global__ void __launch_bounds__(kThreads) step_kernel_noalloc(const __grid_constant__ NoAllocArgs a) {
  using A = typename AccOf<T>::type;
  uint64_t bid = blockIdx.x;
  const int chunk = (int)(bid % (uint64_t)a.nchunks);
  bid /= (uint64_t)a.nchunks;
  const int x = (int)(bid % (uint64_t)a.P);
  const int oi = (int)(bid / (uint64_t)a.P);
  if (oi >= a.nops) return;
  const StepOp op = a.ops[oi];
  const int b = ((x - (int)op.dst_place) % a.P + a.P) % a.P;
  const uint64_t bstart = (uint64_t)b * a.q + ((uint64_t)b < a.rem ? (uint64_t)b : a.rem);
  const uint64_t blen = a.q + ((uint64_t)b < a.rem ? 1 : 0);
  const uint64_t c0 = (uint64_t)chunk * kChunk;
  if (c0 >= blen) return;
  const uint64_t lo = bstart + c0;
  const uint64_t hi = bstart + (blen < c0 + kChunk ? blen : c0 + kChunk);
  const bool has_recv = op.recv_place >= 0;
  const int partner = ((x + a.partner) % a.P + a.P) % a.P;
  const void *recv = has_recv ? na_buf_ptr<A>(a, op.recv_buf, partner) : nullptr;
  void *out0 = na_buf_ptr<A>(a, op.out0_buf, x);
  const void *own0 = na_buf_ptr<A>(a, op.out0_own, x);
  void *out1 = na_buf_ptr<A>(a, op.out1_buf, x);
  const void *own1 = na_buf_ptr<A>(a, op.out1_own, x);

  auto result = [&](const void *own, uint8_t own_buf, uint64_t e, A r) -> A {
    if (!own) return r;
    const A o = load1<T, A>(own_buf, own, e);
    return has_recv ? combine<OP>(o, r) : o;
  };
  auto do1 = [&](uint64_t e) {
    const A r = has_recv ? load1<T, A>(op.recv_buf, recv, e) : A(0);
    const A o0 = result(own0, op.out0_own, e, r);
    const A o1 = out1 ? result(own1, op.out1_own, e, r) : r;
    store1<T, A>(op.out0_buf, out0, e, o0);
    if (out1) store1<T, A>(op.out1_buf, out1, e, o1);
  };
  auto do4 = [&](uint64_t e) {
    A r[4] = {A(0), A(0), A(0), A(0)};
    if (has_recv) load4<T, A>(op.recv_buf, recv, e, r);
    A o0[4], o1[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) o0[k] = o1[k] = r[k];
    if (own0) {
      load4<T, A>(op.out0_own, own0, e, o0);
      if (has_recv)
#pragma unroll
        for (int k = 0; k < 4; ++k) o0[k] = combine<OP>(o0[k], r[k]);
    }
    if (out1 && own1) {
      load4<T, A>(op.out1_own, own1, e, o1);
      if (has_recv)
#pragma unroll
        for (int k = 0; k < 4; ++k) o1[k] = combine<OP>(o1[k], r[k]);
    }
    store4<T, A>(op.out0_buf, out0, e, o0);
    if (out1) store4<T, A>(op.out1_buf, out1, e, o1);
  };
  uint64_t va = (lo + 3) & ~uint64_t(3);
  uint64_t vb = hi & ~uint64_t(3);
  if (va > hi) va = hi;
  if (vb < va) vb = va;
  for (uint64_t e = lo + threadIdx.x; e < va; e += blockDim.x) do1(e);
  for (uint64_t e = va + 4 * (uint64_t)threadIdx.x; e < vb; e += 4 * (uint64_t)blockDim.x) do4(e);
  for (uint64_t e = vb + threadIdx.x; e < hi; e += blockDim.x) do1(e);
}

// Device address of the scratch array on the current device, looked up on every call
// with that device current: the lookup allocates nothing, and a cached address would be
// stale after cudaDeviceReset or in another context on the same device.
int noalloc_scratch(void **out);

}  // namespace

// Loads this file's device code on the current device (and with it the scratch array).
int load_step_module() {
  void *p = nullptr;
  return noalloc_scratch(&p);
}

namespace {

int noalloc_scratch(void **out) {
  void *p = nullptr;
  cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(no-allocation scratch)");
  *out = p;
  return GAR_OK;
}

template <typename T, int OP>
int noalloc_launch(const gar_plan &pl, const Launch &ln, void *const *rank, void *scratch,
                   gar_stream_t stream) {
  NoAllocArgs a{};
  for (int x = 0; x < pl.P; ++x) a.rank[x] = rank[x];
  int slot = 0;
  for (int k = 0; k < NUM_WS_BUFS; ++k) {
    a.ws[k] = pl.ws_used[k] ? static_cast<char *>(scratch) +
                                  (size_t)(slot++) * pl.P * pl.n_pad * acc_size(pl.dtype)
                            : nullptr;
  }
  for (int k = 0; k < ln.nops; ++k) a.ops[k] = pl.ops[ln.first_op + k];
  a.q = pl.q;
  a.rem = pl.rem;
  a.n_pad = pl.n_pad;
  a.P = pl.P;
  a.partner = ln.partner;
  a.nops = ln.nops;
  const uint64_t maxblk = pl.q + (pl.rem ? 1 : 0);
  a.nchunks = (int)((maxblk + kChunk - 1) / kChunk);
  if (a.nchunks == 0 || ln.nops == 0) return GAR_OK;
  const uint64_t grid = (uint64_t)a.nchunks * (uint64_t)pl.P * (uint64_t)ln.nops;
  if (grid > 0x7fffffffull) {
    set_error("no-allocation step launch grid too large");
    return GAR_EINVAL;
  }
  step_kernel_noalloc<T, OP><<<(unsigned)grid, kThreads, 0, (cudaStream_t)stream>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "no-allocation step kernel launch");
  return GAR_OK;
}

template <typename T>
int noalloc_launch_op(const gar_plan &pl, const Launch &ln, void *const *rank, void *scratch,
                      gar_stream_t s) {
  switch (pl.op) {
    case GAR_SUM: return noalloc_launch<T, GAR_SUM>(pl, ln, rank, scratch, s);
    case GAR_MAX: return noalloc_launch<T, GAR_MAX>(pl, ln, rank, scratch, s);
    case GAR_MIN: return noalloc_launch<T, GAR_MIN>(pl, ln, rank, scratch, s);
  }
  return GAR_EINVAL;
}

}  // namespace
}  // namespace gar

extern "C" int gar_allreduce_noalloc(gar_plan *pl, void *const *rank_buffers, gar_stream_t stream) {
  using namespace gar;
  if (pl == nullptr || rank_buffers == nullptr) {
    set_error("null plan or rank buffer array");
    return GAR_EINVAL;
  }
  if (pl->group != GAR_GROUP_CYCLIC) {
    set_error("gar_allreduce_noalloc supports the cyclic group only");
    return GAR_EINVAL;
  }
  if (pl->P > GAR_NOALLOC_MAX_P) {
    set_error("gar_allreduce_noalloc supports P <= " + std::to_string(GAR_NOALLOC_MAX_P) +
              ", plan has P=" + std::to_string(pl->P));
    return GAR_EINVAL;
  }
  if (pl->ws_bytes > (size_t)GAR_NOALLOC_SCRATCH_BYTES) {
    set_error("gar_allreduce_noalloc: plan needs " + std::to_string(pl->ws_bytes) +
              " bytes of workspace, the fixed scratch array holds " +
              std::to_string((size_t)GAR_NOALLOC_SCRATCH_BYTES));
    return GAR_EINVAL;
  }
  for (int x = 0; x < pl->P; ++x) {
    if (rank_buffers[x] == nullptr) {
      set_error("null rank buffer " + std::to_string(x));
      return GAR_EINVAL;
    }
    if (reinterpret_cast<uintptr_t>(rank_buffers[x]) % 16 != 0) {
      set_error("rank buffer " + std::to_string(x) + " is not 16-byte aligned");
      return GAR_EALIGN;
    }
    for (int y = 0; y < x; ++y)
      if (rank_buffers[y] == rank_buffers[x]) {
        set_error("two ranks share one buffer");
        return GAR_EINVAL;
      }
  }
  for (const Launch &ln : pl->launches)
    if (ln.nops > kNoAllocMaxOps) {
      set_error("gar_allreduce_noalloc: a launch has more block ops than the parameter block holds");
      return GAR_EINVAL;
    }
  if (pl->n == 0 || pl->P == 1) return GAR_OK;
  void *scratch = nullptr;
  int rc = noalloc_scratch(&scratch);
  if (rc) return rc;
  for (const Launch &ln : pl->launches) {
    switch (pl->dtype) {
      case GAR_F32: rc = noalloc_launch_op<float>(*pl, ln, rank_buffers, scratch, stream); break;
      case GAR_BF16: rc = noalloc_launch_op<__nv_bfloat16>(*pl, ln, rank_buffers, scratch, stream); break;
      case GAR_I32: rc = noalloc_launch_op<int>(*pl, ln, rank_buffers, scratch, stream); break;
      default: rc = GAR_EINVAL;
    }
    if (rc) return rc;
  }
  return GAR_OK;
}
