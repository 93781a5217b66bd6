// Code generator for the fused and batched kernels.
//
// A plan's fused program (plan.cpp) is a short straight-line list of combines per
// element position.  Emitting it as straight-line CUDA C and compiling it for sm_103a
// at plan creation (jit.cpp) keeps every contribution and partial result in registers
// with compile-time indices, for any P and any step count, instead of interpreting the
// schedule from a table at run time.  The fixed parts of the kernels (vector loads
// and stores, bf16 handling, grid-stride loops) are the text in kSkeleton below.
#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <functional>
#include <map>
#include <stdexcept>
#include <string>
#include <vector>

#include "gar_internal.hpp"

namespace gar {
namespace {

// Types, operators and 1..16-byte vector loads/stores shared by every generated kernel.
// Loads and stores use the streaming cache hints (.cs): every byte is touched once.
const char *kSkeleton = R"CUDA(
typedef unsigned short gar_u16;
typedef unsigned int gar_u32;
typedef unsigned long long gar_u64;

#if GAR_DTYPE == 1
typedef float gar_acc;
typedef gar_u16 gar_io;
#elif GAR_DTYPE == 2
typedef int gar_acc;
typedef int gar_io;
#else
typedef float gar_acc;
typedef float gar_io;
#endif

static __device__ __forceinline__ gar_acc gar_op(gar_acc a, gar_acc b) {
#if GAR_DTYPE == 2
#if GAR_OP == 0
  return (int)((gar_u32)a + (gar_u32)b);
#elif GAR_OP == 1
  return a > b ? a : b;
#else
  return a < b ? a : b;
#endif
#else
#if GAR_OP == 0
  return a + b;
#elif GAR_OP == 1
  return fmaxf(a, b);
#else
  return fminf(a, b);
#endif
#endif
}

// out[w] = a[w] (+) b[w] for W element positions; float sums of an even W pair the
// positions in paired fp32 adds (__fadd2_rn: round to nearest even in each half)
template <int W>
static __device__ __forceinline__ void gar_comb(gar_acc *out, const gar_acc *a, const gar_acc *b) {
#if GAR_DTYPE != 2 && GAR_OP == 0 && GAR_FADD2
  if (W % 2 == 0) {
#pragma unroll
    for (int w = 0; w < W; w += 2) {
      const float2 r = __fadd2_rn(make_float2(a[w], a[w + 1]), make_float2(b[w], b[w + 1]));
      out[w] = r.x;
      out[w + 1] = r.y;
    }
    return;
  }
#endif
#pragma unroll
  for (int w = 0; w < W; ++w) out[w] = gar_op(a[w], b[w]);
}

static __device__ __forceinline__ float gar_bf16_lo(gar_u32 u) { return __uint_as_float(u << 16); }
static __device__ __forceinline__ float gar_bf16_hi(gar_u32 u) { return __uint_as_float(u & 0xffff0000u); }
static __device__ __forceinline__ gar_u32 gar_pack_bf16(float lo, float hi) {
  gar_u32 r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// Load W consecutive elements at p (aligned to W elements) into v[0..W).
template <int W> static __device__ __forceinline__ void gar_load(const gar_io *p, gar_acc *v);
template <int W> static __device__ __forceinline__ void gar_store(gar_io *p, const gar_acc *v);

#if GAR_DTYPE == 1
template <> __device__ __forceinline__ void gar_load<1>(const gar_io *p, gar_acc *v) {
  gar_u16 h;
  asm("ld.global" GAR_LDH ".u16 %0, [%1];" : "=h"(h) : "l"(p));
  v[0] = __uint_as_float(((gar_u32)h) << 16);
}
template <> __device__ __forceinline__ void gar_load<2>(const gar_io *p, gar_acc *v) {
  gar_u32 u;
  asm("ld.global" GAR_LDH ".u32 %0, [%1];" : "=r"(u) : "l"(p));
  v[0] = gar_bf16_lo(u); v[1] = gar_bf16_hi(u);
}
template <> __device__ __forceinline__ void gar_load<4>(const gar_io *p, gar_acc *v) {
  gar_u32 a, b;
  asm("ld.global" GAR_LDH ".v2.u32 {%0,%1}, [%2];" : "=r"(a), "=r"(b) : "l"(p));
  v[0] = gar_bf16_lo(a); v[1] = gar_bf16_hi(a); v[2] = gar_bf16_lo(b); v[3] = gar_bf16_hi(b);
}
template <> __device__ __forceinline__ void gar_load<8>(const gar_io *p, gar_acc *v) {
  gar_u32 a, b, c, d;
  asm("ld.global" GAR_LDH ".v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(a), "=r"(b), "=r"(c), "=r"(d) : "l"(p));
  v[0] = gar_bf16_lo(a); v[1] = gar_bf16_hi(a); v[2] = gar_bf16_lo(b); v[3] = gar_bf16_hi(b);
  v[4] = gar_bf16_lo(c); v[5] = gar_bf16_hi(c); v[6] = gar_bf16_lo(d); v[7] = gar_bf16_hi(d);
}
template <> __device__ __forceinline__ void gar_store<1>(gar_io *p, const gar_acc *v) {
  gar_u16 h;
  asm("cvt.rn.bf16.f32 %0, %1;" : "=h"(h) : "f"(v[0]));
  asm volatile("st.global" GAR_STH ".u16 [%0], %1;" :: "l"(p), "h"(h) : "memory");
}
template <> __device__ __forceinline__ void gar_store<2>(gar_io *p, const gar_acc *v) {
  asm volatile("st.global" GAR_STH ".u32 [%0], %1;" :: "l"(p), "r"(gar_pack_bf16(v[0], v[1])) : "memory");
}
template <> __device__ __forceinline__ void gar_store<4>(gar_io *p, const gar_acc *v) {
  asm volatile("st.global" GAR_STH ".v2.u32 [%0], {%1,%2};" :: "l"(p),
               "r"(gar_pack_bf16(v[0], v[1])), "r"(gar_pack_bf16(v[2], v[3])) : "memory");
}
template <> __device__ __forceinline__ void gar_store<8>(gar_io *p, const gar_acc *v) {
  asm volatile("st.global" GAR_STH ".v4.u32 [%0], {%1,%2,%3,%4};" :: "l"(p),
               "r"(gar_pack_bf16(v[0], v[1])), "r"(gar_pack_bf16(v[2], v[3])),
               "r"(gar_pack_bf16(v[4], v[5])), "r"(gar_pack_bf16(v[6], v[7])) : "memory");
}
#else
template <> __device__ __forceinline__ void gar_load<1>(const gar_io *p, gar_acc *v) {
  gar_u32 a;
  asm("ld.global" GAR_LDH ".b32 %0, [%1];" : "=r"(a) : "l"(p));
  v[0] = *reinterpret_cast<gar_acc *>(&a);
}
template <> __device__ __forceinline__ void gar_load<2>(const gar_io *p, gar_acc *v) {
  gar_u32 a, b;
  asm("ld.global" GAR_LDH ".v2.b32 {%0,%1}, [%2];" : "=r"(a), "=r"(b) : "l"(p));
  v[0] = *reinterpret_cast<gar_acc *>(&a); v[1] = *reinterpret_cast<gar_acc *>(&b);
}
template <> __device__ __forceinline__ void gar_load<4>(const gar_io *p, gar_acc *v) {
  gar_u32 a, b, c, d;
  asm("ld.global" GAR_LDH ".v4.b32 {%0,%1,%2,%3}, [%4];" : "=r"(a), "=r"(b), "=r"(c), "=r"(d) : "l"(p));
  v[0] = *reinterpret_cast<gar_acc *>(&a); v[1] = *reinterpret_cast<gar_acc *>(&b);
  v[2] = *reinterpret_cast<gar_acc *>(&c); v[3] = *reinterpret_cast<gar_acc *>(&d);
}
template <> __device__ __forceinline__ void gar_store<1>(gar_io *p, const gar_acc *v) {
  asm volatile("st.global" GAR_STH ".b32 [%0], %1;" :: "l"(p), "r"(*reinterpret_cast<const gar_u32 *>(&v[0])) : "memory");
}
template <> __device__ __forceinline__ void gar_store<2>(gar_io *p, const gar_acc *v) {
  asm volatile("st.global" GAR_STH ".v2.b32 [%0], {%1,%2};" :: "l"(p),
               "r"(*reinterpret_cast<const gar_u32 *>(&v[0])),
               "r"(*reinterpret_cast<const gar_u32 *>(&v[1])) : "memory");
}
template <> __device__ __forceinline__ void gar_store<4>(gar_io *p, const gar_acc *v) {
  asm volatile("st.global" GAR_STH ".v4.b32 [%0], {%1,%2,%3,%4};" :: "l"(p),
               "r"(*reinterpret_cast<const gar_u32 *>(&v[0])),
               "r"(*reinterpret_cast<const gar_u32 *>(&v[1])),
               "r"(*reinterpret_cast<const gar_u32 *>(&v[2])),
               "r"(*reinterpret_cast<const gar_u32 *>(&v[3])) : "memory");
}
#endif
)CUDA";

// Optional tuning knobs for launch-shape sweeps, read from the environment; each only
// changes how the same work is laid out (never what is computed), and the chosen values
// are part of the generated source, so kernels of different settings never share a cache
// entry.  GAR_TUNE_FUSED_W: elements per thread-vector; GAR_TUNE_FUSED_MINB: minimum
// resident CTAs per SM in __launch_bounds__; GAR_TUNE_LDH / GAR_TUNE_STH: cache-hint
// suffix of the global loads / stores (default ".cs", streaming); GAR_TUNE_DOUBLED (0 or
// 1): whether a rotated cyclic single-thread kernel stores its pointer tables twice;
// GAR_TUNE_BF_ORDER / _BF_WARPS / _BF_MINB: combine order and CTA shape of the
// breadth-first form; GAR_TUNE_SP_PAIR (0: no paired adds, 1: pairs of tracked operand
// pairs, 2: any adjacent placements) / _SP_WARPS / _SP_MINB: the same for the two-lane
// form.
int tune_int(const char *name, int dflt) {
  const char *v = std::getenv(name);
  return (v && *v) ? std::atoi(v) : dflt;
}
std::string tune_str(const char *name, const char *dflt) {
  const char *v = std::getenv(name);
  return (v != nullptr) ? std::string(v) : std::string(dflt);
}

std::string fmt(const char *f, ...) {
  char buf[1024];
  va_list ap;
  va_start(ap, f);
  vsnprintf(buf, sizeof buf, f, ap);
  va_end(ap);
  return std::string(buf);
}

// Emission order of one plan's program: results one after another, each by a
// depth-first walk that evaluates the operand needing more registers first
// (Sethi-Ullman order), contributions loaded at first use, every result's stores
// right after it is complete.
struct Schedule {
  // items: kind 0 = load leaf j, 1 = combine value v, 2 = store result s
  std::vector<std::pair<int, int>> items;
  int peak_live = 0;
};

Schedule order_program(const FusedProgram &fp) {
  const int P = fp.P;
  const int nv = P + (int)fp.a.size();
  std::vector<int> need(nv, 1);
  for (int k = 0; k < (int)fp.a.size(); ++k) {
    const int la = need[fp.a[k]], lb = need[fp.b[k]];
    need[P + k] = la == lb ? la + 1 : std::max(la, lb);
  }
  Schedule sc;
  std::vector<char> done(nv, 0);
  std::function<void(int)> visit = [&](int v) {
    if (done[v]) return;
    if (v < P) {
      sc.items.push_back({0, v});
      done[v] = 1;
      return;
    }
    const int a = fp.a[v - P], b = fp.b[v - P];
    if (need[b] > need[a]) {
      visit(b);
      visit(a);
    } else {
      visit(a);
      visit(b);
    }
    sc.items.push_back({1, v});
    done[v] = 1;
  };
  for (int s = 0; s < fp.K; ++s) {
    visit(fp.out[s]);
    sc.items.push_back({2, s});
  }
  // liveness over this order
  std::vector<int> last_use(nv, -1), def(nv, -1);
  for (int t = 0; t < (int)sc.items.size(); ++t) {
    auto [kind, v] = sc.items[t];
    if (kind == 0) def[v] = t;
    if (kind == 1) {
      def[v] = t;
      last_use[fp.a[v - P]] = t;
      last_use[fp.b[v - P]] = t;
    }
    if (kind == 2) last_use[fp.out[v]] = t;
  }
  std::vector<int> delta(sc.items.size() + 1, 0);
  for (int v = 0; v < nv; ++v) {
    if (def[v] < 0) continue;
    delta[def[v]] += 1;
    delta[std::max(last_use[v], def[v]) + 1] -= 1;
  }
  int live = 0;
  for (int d : delta) {
    live += d;
    sc.peak_live = std::max(sc.peak_live, live);
  }
  return sc;
}

// Largest vector width (elements per thread, at most 16 bytes of input) whose W *
// peak_live values fit the register file without heavy spilling.  Calibrated on GB300
// with P = 127 bf16 at every step count (peak_live 8..254): the fastest width always
// satisfied W * peak_live <= 384, and <= 256 for W = 8; one step past the limit ptxas
// falls back to spilling kilobytes per thread and the kernel runs 2-10x slower.
int choose_width(int dtype, int peak_live, int cap) {
  const int wmax = std::min(cap, 16 / elem_size(dtype));
  int w = wmax;
  while (w > 1 && (w * peak_live > 384 || (w >= 8 && w * peak_live > 256))) w /= 2;
  return w;
}

// Emits `template <int W> gar_eval_<tag>(<params>, u64 e0, int b)`: evaluates the program
// for W consecutive element positions starting at e0, all in block b.  Contribution j is
// read from row ld_row((b + j) mod P) and result placement p is written to row
// st_row((b + p) mod P); with rotate == false the rows are j and p themselves (b = 0).
std::string emit_eval(const FusedProgram &fp, const Schedule &sc, const std::string &tag,
                      const std::string &params,
                      const std::function<std::string(const std::string &)> &ld_row,
                      const std::function<std::string(const std::string &)> &st_row,
                      bool rotate, bool xor_group, bool doubled = false) {
  const int P = fp.P;
  std::string s;
  s += "template <int W>\nstatic __device__ __forceinline__ void gar_eval_" + tag + "(" + params +
       ", gar_u64 e0, int b) {\n";
  s += "  (void)b;\n";
  // rank of contribution / placement j for an element of block b: t_j(b)
  auto rank_of = [&](int j) -> std::string {
    if (!rotate) return std::to_string(j);
    if (j == 0) return "b";
    if (xor_group) return fmt("(b ^ %d)", j);
    // with the pointer tables stored twice, entry b + j (< 2P) is rank (b + j) mod P
    if (doubled) return fmt("(b + %d)", j);
    return fmt("(b + %d >= %d ? b + %d : b + %d)", j, P, j - P, j);
  };
  // stores of result s go to every placement p whose origin is s
  std::vector<std::vector<int>> places(fp.K);
  for (int p = 0; p < P; ++p) places[fp.origin[p]].push_back(p);
  for (auto [kind, v] : sc.items) {
    if (kind == 0) {
      s += fmt("  gar_acc v%d[W]; gar_load<W>(", v) + ld_row(rank_of(v)) + " + e0, v" +
           std::to_string(v) + ");\n";
    } else if (kind == 1) {
      const int a = fp.a[v - P], b = fp.b[v - P];
      s += fmt("  gar_acc v%d[W]; gar_comb<W>(v%d, v%d, v%d);\n",
               v, v, a, b);
    } else {
      const int val = fp.out[v];
      for (int p : places[v])
        s += "  gar_store<W>(" + st_row(rank_of(p)) + " + e0, v" + std::to_string(val) + ");\n";
    }
  }
  s += "}\n";
  return s;
}

std::string dtype_tag(int dtype) { return dtype == GAR_BF16 ? "bf16" : dtype == GAR_I32 ? "i32" : "f32"; }
std::string op_tag(int op) { return op == GAR_MAX ? "max" : op == GAR_MIN ? "min" : "sum"; }

// Block index of element e for a P-way split of n elements (first n mod P blocks one
// longer), with all constants compiled in.
std::string emit_block_of(const std::string &name, int P, uint64_t n) {
  const uint64_t q = n / P, rem = n % P;
  std::string s = "static __device__ __forceinline__ int " + name + "(gar_u64 e) {\n";
  if (q == 0) {
    s += "  return (int)e;\n";
  } else {
    s += fmt("  const gar_u64 big = %lluULL;\n", (unsigned long long)(rem * (q + 1)));
    s += fmt("  return e < big ? (int)(e / %lluULL) : (int)(%lluULL + (e - big) / %lluULL);\n",
             (unsigned long long)(q + 1), (unsigned long long)rem, (unsigned long long)q);
  }
  s += "}\n";
  return s;
}

}  // namespace

CodegenResult generate_fused_source(const gar_plan &pl, int threads_override, int minb_override, int fadd2_override) {
  const FusedProgram &fp = pl.prog;
  const int P = pl.P;
  Schedule sc = order_program(fp);
  const bool rotate = pl.K != P;   // latency-optimal results do not depend on the block
  // Single-copy cyclic programs over 32 or more contributions run in 32-thread CTAs of at
  // most 128 registers, with doubled pointer tables: a thread's P loads take long and
  // vary, and a one-warp CTA frees its slot as soon as that warp is done instead of
  // waiting for the slowest of eight.  GB300, against 256-thread CTAs: P = 127 x 8 MiB
  // bf16 S = 14 0.351 -> 0.322 ms, P = 100 x 8 MiB bf16 0.270 -> 0.253, P = 40 x 12 MiB
  // bf16 0.163 -> 0.151, P = 32 x 32 MiB bf16 0.334 -> 0.312, P = 127 x 8 MiB fp32
  // 0.336 -> 0.327, P = 64 x 16 MiB fp32 0.324 -> 0.318, P = 64 x 16 MiB bf16 unchanged
  // (0.314).  Without the doubled tables the 128-register cap spills (P = 127 bf16:
  // 0.389 ms); fewer contributions gain nothing (P = 24 x 64 MiB fp32 0.467 ms either
  // way) or lose (P = 8 x 256 MiB bf16 0.619 -> 0.627 ms).
  const bool small_cta = pl.K == 1 && P >= 32 && P <= 1000 && rotate && pl.group != GAR_GROUP_XOR;
  bool doubled = rotate && pl.group != GAR_GROUP_XOR && P <= 1000 && (pl.K > 1 || small_cta);
  if (const int d = tune_int("GAR_TUNE_DOUBLED", -1); d >= 0)
    doubled = d != 0 && rotate && pl.group != GAR_GROUP_XOR && P <= 1000;
  // bf16 programs with doubled pointer tables (below) run best with at most 8-byte
  // vectors (P = 127, S = 8..13: W = 8 was 3-6 % slower at S = 12, 13 than W = 4).
  int W = choose_width(pl.dtype, sc.peak_live, (doubled && pl.dtype == GAR_BF16) ? 4 : 16);
  // Few element positions: narrower vectors give more threads, and the contributions'
  // load latencies then overlap across warps instead of queueing in one (P = 127 bf16
  // with 212 positions: 92 us at W = 8, 24 us at W = 1).
  while (W > 1 && pl.n / (uint64_t)W < 16384) W /= 2;
  if (int w = tune_int("GAR_TUNE_FUSED_W", 0))
    if (w > 0 && (w & (w - 1)) == 0 && w * elem_size(pl.dtype) <= 16) W = w;
  const int minb = minb_override > 0 ? minb_override : tune_int("GAR_TUNE_FUSED_MINB", small_cta ? 16 : 0);
  int nthr = threads_override > 0 ? threads_override : tune_int("GAR_TUNE_FUSED_THREADS", small_cta ? 32 : 256);
  if (nthr < 32 || nthr > 1024 || nthr % 32 != 0) nthr = 256;
  const std::string bounds = minb > 0 ? fmt("__launch_bounds__(%d, %d)", nthr, minb)
                                      : fmt("__launch_bounds__(%d)", nthr);
  CodegenResult cg;
  cg.width = W;
  cg.threads = nthr;
  cg.kernel_name = fmt("gar_fused_P%d_S%d_K%d_", P, pl.S, pl.K) + dtype_tag(pl.dtype) + "_" +
                   op_tag(pl.op) + fmt("_W%d", W) + (pl.group == GAR_GROUP_XOR ? "_xor" : "");
  std::string s;
  s += fmt("#define GAR_DTYPE %d\n#define GAR_OP %d\n", pl.dtype, pl.op);
  // paired fp32 adds over element positions for bf16 programs at W >= 4 (P = 127:
  // S = 10 0.377 -> 0.360 ms, S = 11 0.354 -> 0.344 ms); fp32 programs were slower or
  // spilled (P = 64 fp32, S = 8: 104 -> 255 registers); bf16 at W = 2 takes them only
  // through fadd2_override, when the plan's prepared kernel is register-bound anyway
  const int fadd2 = fadd2_override >= 0 ? fadd2_override : tune_int("GAR_TUNE_FADD2", pl.dtype == GAR_BF16 && W >= 4);
  s += fmt("#define GAR_FADD2 %d\n", fadd2 != 0 ? 1 : 0);
  s += "#define GAR_LDH \"" + tune_str("GAR_TUNE_LDH", ".cs") + "\"\n";
  s += "#define GAR_STH \"" + tune_str("GAR_TUNE_STH", ".cs") + "\"\n";
  s += kSkeleton;
  s += fmt("#define GAR_P %d\n#define GAR_W %d\n", P, W);
  s += fmt("#define GAR_N %lluULL\n", (unsigned long long)pl.n);
  // in[] / out[]: where rank x's contributions are read and its results written (equal
  // for the in-place Allreduce); [e_lo, e_hi): the element positions this launch covers
  // (e_lo a multiple of GAR_W), so one Allreduce can run as several launches.
  // Rotated cyclic programs index the pointer tables with (b + j) mod P; storing each
  // table twice turns that into b + j, which folds into the constant-bank offset of the
  // pointer load (the parameter block stays within 32 KB up to P = 1000).  Only for
  // programs with several result copies (K > 1): there it freed registers and made P = 127
  // bf16 up to 19 % faster (S = 8..13).  The single-copy programs (bandwidth-optimal, folds,
  // the Ring) are HBM-bound and mostly ran slower with it: P = 24 x 64 MiB fp32 S = 10 by
  // 0.8 %, P = 24 x 64 MiB bf16 S = 10 by 1.1 %, P = 8 x 256 MiB bf16 S = 6 by 4 %
  // (P = 127 x 8 MiB bf16 S = 14 ran 1 % faster).
  cg.table_copies = doubled ? 2 : 1;
  s += fmt("struct gar_args { const gar_io *in[%d]; gar_io *out[%d]; gar_u64 e_lo, e_hi; };\n",
           cg.table_copies * P, cg.table_copies * P);
  s += emit_block_of("gar_block_of", P, pl.n);
  // When blocks are shorter than a warp's span, the lanes of a warp work on different
  // blocks b, and a rotated program's pointer index (b + j) differs across the warp:
  // indexing the kernel parameters with it serialises (P = 127, 425 B: 34 us against
  // 5.6 us unrotated).  Such kernels first copy the tables to shared memory, where
  // divergent indices are cheap.
  const int tp = cg.table_copies * P;
  const bool staged = rotate && pl.n / (uint64_t)P < 32ull * (uint64_t)W;
  auto ld_row = [staged](const std::string &r) { return (staged ? "tin[" : "a.in[") + r + "]"; };
  auto st_row = [staged](const std::string &r) { return (staged ? "tout[" : "a.out[") + r + "]"; };
  s += emit_eval(fp, sc, "plan",
                 staged ? "const gar_io *const *tin, gar_io *const *tout" : "const gar_args &a", ld_row,
                 st_row, rotate, pl.group == GAR_GROUP_XOR, doubled);
  const std::string ev_args = staged ? "s_in, s_out" : "a";
  s += "extern \"C\" __global__ void " + bounds + " " + cg.kernel_name +
       "(const __grid_constant__ gar_args a) {\n";
  if (staged) {
    s += fmt("  __shared__ const gar_io *s_in[%d];\n  __shared__ gar_io *s_out[%d];\n", tp, tp);
    s += fmt("  for (int i = threadIdx.x; i < %d; i += blockDim.x) { s_in[i] = a.in[i]; s_out[i] = a.out[i]; }\n", tp);
    s += "  __syncthreads();\n";
  }
  // launched with programmatic stream serialisation: nothing is read before every
  // earlier kernel on the stream has completed
  s += "  asm volatile(\"griddepcontrol.wait;\" ::: \"memory\");\n";
  s += "  const gar_u64 v_lo = a.e_lo / GAR_W, v_hi = a.e_hi / GAR_W;\n";
  s += "  const gar_u64 stride = (gar_u64)gridDim.x * blockDim.x;\n";
  s += "  const gar_u64 tid = (gar_u64)blockIdx.x * blockDim.x + threadIdx.x;\n";
  s += "  for (gar_u64 v = v_lo + tid; v < v_hi; v += stride) {\n";
  s += "    const gar_u64 e0 = v * GAR_W;\n";
  if (rotate) {
    s += "    const int b0 = gar_block_of(e0);\n";
    s += "    if (GAR_W == 1 || b0 == gar_block_of(e0 + GAR_W - 1)) {\n";
    s += "      gar_eval_plan<GAR_W>(" + ev_args + ", e0, b0);\n";
    s += "    } else {\n";
    s += "      for (int w = 0; w < GAR_W; ++w) gar_eval_plan<1>(" + ev_args + ", e0 + w, gar_block_of(e0 + w));\n";
    s += "    }\n";
  } else {
    s += "    gar_eval_plan<GAR_W>(" + ev_args + ", e0, 0);\n";
  }
  s += "  }\n";
  s += "  const gar_u64 t0 = (v_hi * GAR_W > a.e_lo ? v_hi * GAR_W : a.e_lo);\n";
  s += "  if (tid < a.e_hi - t0) {\n";
  s += "    const gar_u64 e = t0 + tid;\n";
  s += rotate ? "    gar_eval_plan<1>(" + ev_args + ", e, gar_block_of(e));\n"
              : "    gar_eval_plan<1>(" + ev_args + ", e, 0);\n";
  s += "  }\n";
  s += "  asm volatile(\"griddepcontrol.launch_dependents;\" ::: \"memory\");\n}\n";
  cg.source = s;
  return cg;
}

// ---------------------------------------------------------------------------
// Breadth-first fused kernel, for programs whose single-thread form is register-bound.
//
// With many result copies the schedule keeps a q' and a q* vector at most placements
// (Sec. "Latency-optimal version"): at P = 127, S = 7 about 2P = 254 values per element
// position are alive at once, the kernel above spills and runs one 256-thread CTA per
// SM.  This form evaluates the same program step by step instead of result by result:
//  * every contribution is loaded at the start, so a warp waits for memory once;
//  * the combines of one step (which never depend on each other) follow in placement
//    order, which leaves the compiler long independent runs to schedule;
//  * in float sums, two combines whose placements, operands and results form adjacent
//    pairs run as one paired fp32 add (__fadd2_rn: round to nearest even in each half);
//  * bf16 contributions enter a sum through the mixed-precision add.rn.f32.bf16 (the
//    bf16 value widens exactly, one rounding), so they are never unpacked separately;
//  * small CTAs (32 or 64 threads), several per SM, so the CTAs of an SM drift apart and
//    one's loads overlap another's combines.
// Both adds round exactly as the scalar fp32 add does, so the bits are the schedule's.
// ---------------------------------------------------------------------------

namespace {

const char *kBFHelpers = R"CUDA(
static __device__ __forceinline__ gar_acc gar_wide(gar_io x) {
#if GAR_DTYPE == 1
  return __uint_as_float(((gar_u32)x) << 16);
#else
  return x;
#endif
}
static __device__ __forceinline__ gar_io gar_ldio(const gar_io *p) {
  gar_io v;
#if GAR_DTYPE == 1
  asm volatile("ld.global" GAR_LDH ".u16 %0, [%1];" : "=h"(v) : "l"(p));
#elif GAR_DTYPE == 2
  asm volatile("ld.global" GAR_LDH ".b32 %0, [%1];" : "=r"(v) : "l"(p));
#else
  asm volatile("ld.global" GAR_LDH ".f32 %0, [%1];" : "=f"(v) : "l"(p));
#endif
  return v;
}
static __device__ __forceinline__ void gar_stio(gar_io *p, gar_acc v) {
#if GAR_DTYPE == 1
  gar_u16 h;
  asm("cvt.rn.bf16.f32 %0, %1;" : "=h"(h) : "f"(v));
  asm volatile("st.global" GAR_STH ".u16 [%0], %1;" :: "l"(p), "h"(h) : "memory");
#elif GAR_DTYPE == 2
  asm volatile("st.global" GAR_STH ".b32 [%0], %1;" :: "l"(p), "r"(v) : "memory");
#else
  asm volatile("st.global" GAR_STH ".f32 [%0], %1;" :: "l"(p), "f"(v) : "memory");
#endif
}
#if GAR_DTYPE == 1 && GAR_OP == 0
// (widened bf16 h) + c with one rounding: the fp32 sum of the exactly widened value
static __device__ __forceinline__ float gar_addbf(gar_u16 h, float c) {
  float r;
  asm("add.rn.f32.bf16 %0, %1, %2;" : "=f"(r) : "h"(h), "f"(c));
  return r;
}
#endif
)CUDA";

}  // namespace

int fused_peak_live(const gar_plan &pl) { return order_program(pl.prog).peak_live; }

CodegenResult generate_fused_bf_source(const gar_plan &pl) {
  const FusedProgram &fp = pl.prog;
  const int P = pl.P;
  const int nc = (int)fp.a.size();
  const int nv = P + nc;
  if ((int)fp.place.size() != nc || (int)fp.star.size() != nc)
    throw std::logic_error("fused program without placements");
  const bool rotate = pl.K != P;
  const bool xr = pl.group == GAR_GROUP_XOR;
  const bool sum_f = pl.op == GAR_SUM && pl.dtype != GAR_I32;
  const bool bf16_sum = pl.op == GAR_SUM && pl.dtype == GAR_BF16;

  // level of a value: the step that creates it (contributions: 0); combines by level
  std::vector<int> level(nv, 0);
  int maxlvl = 0;
  for (int k = 0; k < nc; ++k) {
    level[P + k] = 1 + std::max(level[fp.a[k]], level[fp.b[k]]);
    maxlvl = std::max(maxlvl, level[P + k]);
  }
  // order of a level's combines: 0 as built (the q* of a step, then its q'), 1 by
  // placement with q' first, 2 by placement with q* first (GAR_TUNE_BF_ORDER)
  const int order = tune_int("GAR_TUNE_BF_ORDER", 2);
  std::vector<std::vector<int>> comb(maxlvl + 1);
  for (int k = 0; k < nc; ++k) comb[level[P + k]].push_back(k);
  if (order != 0)
    for (auto &cl : comb)
      std::stable_sort(cl.begin(), cl.end(), [&](int x, int y) {
        if (fp.place[x] != fp.place[y]) return fp.place[x] < fp.place[y];
        return order == 1 ? fp.star[x] < fp.star[y] : fp.star[x] > fp.star[y];
      });
  std::vector<char> needs_leaf(P, 0);
  for (int k = 0; k < nc; ++k)
    for (int x : {fp.a[k], fp.b[k]})
      if (x < P) needs_leaf[x] = 1;
  for (int v : fp.out)
    if (v < P) needs_leaf[v] = 1;

  // Paired adds: combines (c1, c2) of one level whose operands are the low and high
  // halves of pairs, in that order; their results become a pair.  Results at placements
  // 2k and 2k + 1 of the same kind (q' or q*) also form a pair for later levels when
  // they were computed one by one.  fp32 contributions pair as 2k, 2k + 1; bf16 ones go
  // through the mixed add instead.
  std::vector<int> pair_hi(nv, -1), mate(nc, -1);
  std::vector<char> is_hi(nc, 0), hi_taken(nv, 0);
  if (sum_f) {
    std::map<std::pair<int, int>, int> by_ops;
    for (int k = 0; k < nc; ++k) by_ops[{fp.a[k], fp.b[k]}] = k;
    if (pl.dtype == GAR_F32)
      for (int j = 0; j + 1 < P; j += 2) {
        pair_hi[j] = j + 1;
        hi_taken[j + 1] = 1;
      }
    for (int L = 1; L <= maxlvl; ++L) {
      const std::vector<int> &cl = comb[L];
      for (int c1 : cl) {
        if (mate[c1] >= 0 || is_hi[c1]) continue;
        const int ha = pair_hi[fp.a[c1]], hb = pair_hi[fp.b[c1]];
        if (ha < 0 || hb < 0) continue;
        auto it = by_ops.find({ha, hb});
        if (it == by_ops.end()) continue;
        const int c2 = it->second;
        if (c2 == c1 || mate[c2] >= 0 || is_hi[c2] || level[P + c2] != L) continue;
        mate[c1] = c2;
        is_hi[c2] = 1;
        pair_hi[P + c1] = P + c2;
        hi_taken[P + c2] = 1;
      }
      std::map<std::pair<int, int>, int> at;  // (placement, star) -> value
      for (int c : cl) at[{fp.place[c], fp.star[c]}] = P + c;
      for (int c : cl) {
        const int v = P + c;
        if (fp.place[c] % 2 != 0 || pair_hi[v] >= 0 || is_hi[c]) continue;
        auto it = at.find({fp.place[c] + 1, fp.star[c]});
        if (it == at.end() || hi_taken[it->second] || pair_hi[it->second] >= 0) continue;
        pair_hi[v] = it->second;
        hi_taken[it->second] = 1;
      }
    }
  }

  // Launch shape, from P = 127 x 8 MiB bf16 on GB300: 168 registers (a third warp per
  // sub-partition register file) in 128-thread CTAs, 3 per SM (S = 8, 192 live values:
  // 0.464 ms; 0.473 ms in 64-thread CTAs, 0.48 ms in 32-thread ones, 0.56-0.60 ms at 255
  // or 128 registers).  The widest programs (S = 7, 254 live values) evaluate their
  // results in two passes (below), which brings them to 168 registers too: 0.552 ms,
  // against 0.600 ms in one pass at 255 registers in 32-thread CTAs, 8 per SM.
  const int peak = order_program(fp).peak_live;
  const bool widest = peak >= 224;
  const int warps = std::max(1, std::min(16, tune_int("GAR_TUNE_BF_WARPS", 4)));
  const int minb = std::max(1, tune_int("GAR_TUNE_BF_MINB", 3));
  // The results in G passes over contiguous groups of result copies, each pass evaluating
  // only the values its group's results depend on: shared values are computed again in
  // every pass that needs them, for fewer values alive at once.  The first pass copies the
  // contributions to shared memory, where later passes read them (the first pass's
  // results may already have overwritten them in place).  P = 127, S = 7: 1752
  // combines in two passes instead of 1524, about 190 values alive instead of 286.
  // S = 8 (64 copies) lost: 996 combines in two passes, 158 values alive instead of 190,
  // 0.477-0.516 ms against 0.464 in one.  GAR_TUNE_BF_GROUPS overrides G.
  const int groups = std::max(1, std::min(fp.K, tune_int("GAR_TUNE_BF_GROUPS", widest ? 2 : 1)));
  // Pointer tables: the kernel parameters, indexed b + j (stored twice), while a warp's
  // 32 element positions share one block almost always (blocks of 32+ elements); with
  // shorter blocks the index differs across the lanes and the tables go to shared memory.
  const bool smem_tab = rotate && pl.n / (uint64_t)P < 32;
  const int tp = (rotate && !xr) ? 2 * P : P;
  CodegenResult cg;
  cg.width = 1;
  cg.table_copies = (rotate && !xr) ? 2 : 1;
  cg.threads = 32 * warps;
  cg.form = 1;
  cg.kernel_name = fmt("gar_fusedbf_P%d_S%d_K%d_", P, pl.S, pl.K) + dtype_tag(pl.dtype) + "_" +
                   op_tag(pl.op) + (xr ? "_xor" : "");

  std::string s;
  s += fmt("#define GAR_DTYPE %d\n#define GAR_OP %d\n", pl.dtype, pl.op);
  s += "#define GAR_LDH \"" + tune_str("GAR_TUNE_LDH", ".cs") + "\"\n";
  s += "#define GAR_STH \"" + tune_str("GAR_TUNE_STH", ".cs") + "\"\n";
  s += kSkeleton;
  s += kBFHelpers;
  s += fmt("struct gar_args { const gar_io *in[%d]; gar_io *out[%d]; gar_u64 e_lo, e_hi; };\n",
           cg.table_copies * P, cg.table_copies * P);
  if (rotate) s += emit_block_of("gar_block_of", P, pl.n);

  // contribution j of an element of block b comes from rank t_j(b); result placement p
  // goes to rank t_p(b) (latency-optimal programs: no rotation, b = 0)
  auto rank_of = [&](int j) -> std::string {
    if (!rotate) return std::to_string(j);
    if (j == 0) return "b";
    return xr ? fmt("(b ^ %d)", j) : fmt("(b + %d)", j);
  };
  const std::string tin = smem_tab ? "tin[" : "a.in[", tout = smem_tab ? "tout[" : "a.out[";
  std::string f = "static __device__ __forceinline__ void gar_eval_bf(const gar_args &a, ";
  f += smem_tab ? "const gar_io *const *tin, gar_io *const *tout, " : "";
  f += "gar_u64 e, int b) {\n  (void)a; (void)b;\n";
  if (groups > 1) {
    s += fmt("#define GAR_BF_THREADS %d\n", cg.threads);
    f += fmt("  __shared__ gar_io gar_sl_all[%d * GAR_BF_THREADS];\n", P);
    f += "  gar_io *const gar_sl = gar_sl_all + threadIdx.x;\n";
  }
  std::vector<int> lo_of(nc, -1);
  for (int k = 0; k < nc; ++k)
    if (mate[k] >= 0) lo_of[mate[k]] = k;
  std::vector<std::vector<int>> places_of(fp.K);
  for (int p = 0; p < P; ++p) places_of[fp.origin[p]].push_back(p);
  for (int g = 0; g < groups; ++g) {
    // group g: result copies [c_lo, c_hi), each stored to every placement that holds it
    const int c_lo = g * fp.K / groups, c_hi = (g + 1) * fp.K / groups;
    std::vector<char> in_cone(nv, groups == 1 ? 1 : 0);
    if (groups > 1) {
      std::vector<int> st;
      for (int sc = c_lo; sc < c_hi; ++sc) st.push_back(fp.out[sc]);
      while (!st.empty()) {
        const int v = st.back();
        st.pop_back();
        if (in_cone[v]) continue;
        in_cone[v] = 1;
        if (v >= P) {
          st.push_back(fp.a[v - P]);
          st.push_back(fp.b[v - P]);
        }
      }
    }
    const std::string sfx = g == 0 ? "" : fmt("_%d", g);
    // the first pass loads every contribution (later passes read its shared-memory copy)
    for (int j = 0; j < P; ++j)
      if (needs_leaf[j] && (in_cone[j] || g == 0))
        f += g == 0 ? fmt("  const gar_io l%d", j) + sfx + " = gar_ldio(" + tin + rank_of(j) + "] + e);\n"
                    : fmt("  const gar_io l%d", j) + sfx + fmt(" = gar_sl[%d * GAR_BF_THREADS];\n", j);
    if (g == 0 && groups > 1)
      for (int j = 0; j < P; ++j)
        if (needs_leaf[j]) f += fmt("  gar_sl[%d * GAR_BF_THREADS] = l%d;\n", j, j);
    auto opnd = [&](int x) { return (x < P ? fmt("gar_wide(l%d", x) + sfx + ")" : fmt("v%d", x) + sfx); };
    auto nm = [&](const char *f0, int v) { return fmt(f0, v) + sfx; };
    for (int L = 1; L <= maxlvl; ++L) {
      for (int k : comb[L]) {
        const int v = P + k, a = fp.a[k], b = fp.b[k];
        if (!in_cone[v]) continue;
        if (is_hi[k] && in_cone[P + lo_of[k]]) continue;
        if (mate[k] >= 0 && in_cone[P + mate[k]]) {
          const int k2 = mate[k], v2 = P + k2;
          f += "  const float2 " + nm("w%d", v) + " = __fadd2_rn(make_float2(" + opnd(a) + ", " + opnd(fp.a[k2]) +
               "), make_float2(" + opnd(b) + ", " + opnd(fp.b[k2]) + "));\n";
          f += "  const gar_acc " + nm("v%d", v) + " = " + nm("w%d", v) + ".x, " + nm("v%d", v2) + " = " +
               nm("w%d", v) + ".y;\n";
        } else if (bf16_sum && (a < P || b < P)) {
          const int lf = a < P ? a : b, other = a < P ? b : a;
          f += "  const gar_acc " + nm("v%d", v) + " = gar_addbf(" + nm("l%d", lf) + ", " + opnd(other) + ");\n";
        } else {
          f += "  const gar_acc " + nm("v%d", v) + " = gar_op(" + opnd(a) + ", " + opnd(b) + ");\n";
        }
      }
    }
    for (int sc = c_lo; sc < c_hi; ++sc)
      for (int p : places_of[sc]) f += "  gar_stio(" + tout + rank_of(p) + "] + e, " + opnd(fp.out[sc]) + ");\n";
  }
  f += "}\n";
  s += f;

  s += fmt("extern \"C\" __global__ void __launch_bounds__(%d, %d) ", cg.threads, minb) + cg.kernel_name +
       "(const __grid_constant__ gar_args a) {\n";
  if (smem_tab) {
    s += fmt("  __shared__ const gar_io *s_in[%d];\n  __shared__ gar_io *s_out[%d];\n", tp, tp);
    s += fmt("  for (int i = threadIdx.x; i < %d; i += blockDim.x) { s_in[i] = a.in[i]; s_out[i] = a.out[i]; }\n", tp);
    s += "  __syncthreads();\n";
  }
  // launched with programmatic stream serialisation: nothing is read before every
  // earlier kernel on the stream has completed
  s += "  asm volatile(\"griddepcontrol.wait;\" ::: \"memory\");\n";
  s += "  const gar_u64 npos = a.e_hi - a.e_lo;\n";
  s += "  const gar_u64 stride = (gar_u64)gridDim.x * blockDim.x;\n";
  // one element position per thread
  s += "  for (gar_u64 i = (gar_u64)blockIdx.x * blockDim.x + threadIdx.x; i < npos; i += stride) {\n";
  s += "    const gar_u64 e = a.e_lo + i;\n";
  s += rotate ? "    const int b = gar_block_of(e);\n" : "    const int b = 0;\n";
  s += std::string("    gar_eval_bf(a, ") + (smem_tab ? "s_in, s_out, " : "") + "e, b);\n";
  s += "  }\n";
  s += "  asm volatile(\"griddepcontrol.launch_dependents;\" ::: \"memory\");\n}\n";
  cg.source = s;
  return cg;
}


// ---------------------------------------------------------------------------
// Two-lane fused kernel for latency-optimal cyclic programs (K = P).
//
// The latency-optimal schedule keeps a q' and a q* vector at every placement (Sec.
// "Latency-optimal version"): about 2P values per element position, which holds the
// one-thread forms at 255 registers and spills.  Here two lanes of a warp share an
// element position, lanes 0-15 and 16-31 of a warp serving the same 16 positions:
//  * lane half A evaluates every combine at placements [0, m), m = ceil(P / 2), and
//    half B the same code rotated by m placements, i.e. placements m .. m + m - 1 (mod
//    P).  The program is invariant under rotation (copy s of the schedule is copy 0
//    shifted by s), so one instruction stream serves both halves; for odd P the
//    halves overlap in one placement, which B computes but does not store;
//  * a step's shift by d moves some vectors across the halves' boundary.  Such an
//    operand comes from the other half by one warp shuffle (xor 16): for the value A
//    needs at placement g >= m, B holds it as its own value at g - m; B's counterpart
//    is A's value at g - m + 1 (odd P) or g - m (even P).  Each half puts the value
//    the other needs into the shuffle, so one shuffle serves both;
//  * contributions and results go through pointer tables in shared memory indexed
//    from each half's rank offset.
// The combines and their operands are the schedule's, so the bits are too.
// ---------------------------------------------------------------------------

namespace {

const char *kSplitHelpers = R"CUDA(
static __device__ __forceinline__ gar_acc gar_xacc(gar_acc v) { return __shfl_xor_sync(0xffffffffu, v, 16); }
static __device__ __forceinline__ gar_io gar_xio(gar_io v) {
#if GAR_DTYPE == 1
  return (gar_io)__shfl_xor_sync(0xffffffffu, (unsigned)v, 16);
#else
  return __shfl_xor_sync(0xffffffffu, v, 16);
#endif
}
)CUDA";

}  // namespace

bool split_form_applies(const gar_plan &pl) {
  const FusedProgram &fp = pl.prog;
  const int P = pl.P;
  if (pl.K != P || P < 4 || P > 1000 || pl.group == GAR_GROUP_XOR) return false;
  const int nc = (int)fp.a.size();
  if ((int)fp.place.size() != nc || (int)fp.star.size() != nc) return false;
  // rotation by one placement maps the program onto itself
  std::map<std::pair<int, int>, int> by_ops;
  for (int k = 0; k < nc; ++k) by_ops[{fp.a[k], fp.b[k]}] = k;
  std::vector<int> rot(P + nc, -1);
  for (int j = 0; j < P; ++j) rot[j] = (j + 1) % P;
  for (int k = 0; k < nc; ++k) {
    const int ra = rot[fp.a[k]], rb = rot[fp.b[k]];
    if (ra < 0 || rb < 0) return false;
    auto it = by_ops.find({ra, rb});
    if (it == by_ops.end() || fp.place[it->second] != (fp.place[k] + 1) % P ||
        fp.star[it->second] != fp.star[k])
      return false;
    rot[P + k] = P + it->second;
  }
  for (int p = 0; p < P; ++p) {
    const int v = fp.out[fp.origin[p]];
    if (v < P || fp.place[v - P] != p) return false;
  }
  return true;
}

CodegenResult generate_fused_split_source(const gar_plan &pl) {
  if (!split_form_applies(pl)) throw std::logic_error("program is not rotation invariant");
  const FusedProgram &fp = pl.prog;
  const int P = pl.P;
  const int nc = (int)fp.a.size();
  const int nv = P + nc;
  const int m = (P + 1) / 2;
  const bool odd = P % 2 == 1;
  const bool sum_f = pl.op == GAR_SUM && pl.dtype != GAR_I32;
  const bool bf16_sum = pl.op == GAR_SUM && pl.dtype == GAR_BF16;
  auto plc = [&](int v) { return v < P ? v : (int)fp.place[v - P]; };

  // rotations of every value by r placements, r = 1 .. P - 1 as needed
  std::map<std::pair<int, int>, int> by_ops;
  for (int k = 0; k < nc; ++k) by_ops[{fp.a[k], fp.b[k]}] = k;
  auto rotation = [&](int r) {
    std::vector<int> rt(nv);
    for (int j = 0; j < P; ++j) rt[j] = (j + r) % P;
    for (int k = 0; k < nc; ++k) rt[P + k] = P + by_ops.at({rt[fp.a[k]], rt[fp.b[k]]});
    return rt;
  };
  const std::vector<int> rot_b = rotation(P - m);                 // what B sends: g - m
  const std::vector<int> rot_a = rotation(odd ? P - m + 1 : P - m);  // what A sends

  std::vector<int> level(nv, 0);
  int maxlvl = 0;
  for (int k = 0; k < nc; ++k) {
    level[P + k] = 1 + std::max(level[fp.a[k]], level[fp.b[k]]);
    maxlvl = std::max(maxlvl, level[P + k]);
  }
  // half A's combines, by level, in placement order (q* first at one placement)
  std::vector<std::vector<int>> comb(maxlvl + 1);
  for (int k = 0; k < nc; ++k)
    if (fp.place[k] < m) comb[level[P + k]].push_back(k);
  for (auto &cl : comb)
    std::stable_sort(cl.begin(), cl.end(), [&](int x, int y) {
      if (fp.place[x] != fp.place[y]) return fp.place[x] < fp.place[y];
      return fp.star[x] > fp.star[y];
    });

  // Paired adds (float sums): two combines of a level at adjacent placements, same
  // kind, whose operands are pairs in the same order, run as one __fadd2_rn.  Pairs:
  // fp32 contributions 2k, 2k + 1; the results of a paired add; results at placements
  // 2k, 2k + 1 of one kind; values received from the other half for such pairs.
  const int pair_mode = tune_int("GAR_TUNE_SP_PAIR", 1);
  std::vector<int> pair_hi(nv, -1), mate(nc, -1);
  std::vector<char> is_hi(nc, 0);
  if (sum_f && pair_mode > 0) {
    if (pl.dtype == GAR_F32)
      for (int j = 0; j + 1 < P; j += 2) pair_hi[j] = j + 1;
    for (int L = 1; L <= maxlvl; ++L) {
      const std::vector<int> &cl = comb[L];
      std::map<std::pair<int, int>, int> at;  // (placement, star) -> combine
      for (int c : cl) at[{fp.place[c], fp.star[c]}] = c;
      for (int c1 : cl) {
        if (mate[c1] >= 0 || is_hi[c1]) continue;
        auto it = at.find({fp.place[c1] + 1, fp.star[c1]});
        if (it == at.end()) continue;
        const int c2 = it->second;
        if (mate[c2] >= 0 || is_hi[c2] || fp.place[c2] >= m) continue;
        const int a1 = fp.a[c1], b1 = fp.b[c1], a2 = fp.a[c2], b2 = fp.b[c2];
        const bool leafbf = bf16_sum && (a1 < P || b1 < P || a2 < P || b2 < P);
        if (leafbf) continue;
        const bool ok = pair_mode == 2 || (pair_hi[a1] == a2 && pair_hi[b1] == b2);
        if (!ok) continue;
        mate[c1] = c2;
        is_hi[c2] = 1;
        pair_hi[P + c1] = P + c2;
      }
      for (int c : cl) {
        const int v = P + c;
        if (fp.place[c] % 2 != 0 || pair_hi[v] >= 0 || is_hi[c]) continue;
        auto it = at.find({fp.place[c] + 1, fp.star[c]});
        if (it == at.end() || is_hi[it->second] || pair_hi[P + it->second] >= 0) continue;
        pair_hi[v] = P + it->second;
      }
    }
  }

  const int warps = std::max(1, std::min(16, tune_int("GAR_TUNE_SP_WARPS", 4)));
  const int minb = std::max(1, tune_int("GAR_TUNE_SP_MINB", 3));
  CodegenResult cg;
  cg.width = 1;
  cg.table_copies = 2;
  cg.threads = 32 * warps;
  cg.form = 2;
  cg.kernel_name = fmt("gar_fusedsp_P%d_S%d_K%d_", P, pl.S, pl.K) + dtype_tag(pl.dtype) + "_" + op_tag(pl.op);

  std::string s;
  s += fmt("#define GAR_DTYPE %d\n#define GAR_OP %d\n", pl.dtype, pl.op);
  s += "#define GAR_LDH \"" + tune_str("GAR_TUNE_LDH", ".cs") + "\"\n";
  s += "#define GAR_STH \"" + tune_str("GAR_TUNE_STH", ".cs") + "\"\n";
  s += kSkeleton;
  s += kBFHelpers;
  s += kSplitHelpers;
  s += fmt("struct gar_args { const gar_io *in[%d]; gar_io *out[%d]; gar_u64 e_lo, e_hi; };\n", 2 * P, 2 * P);

  std::string f = "static __device__ __forceinline__ void gar_eval_sp(const gar_io *const *tin, "
                  "gar_io *const *tout, gar_u64 e, int hb, bool ok) {\n  (void)hb;\n";
  std::vector<char> need_leaf(P, 0);
  for (int L = 1; L <= maxlvl; ++L)
    for (int k : comb[L])
      for (int x : {fp.a[k], fp.b[k]})
        if (x < P) need_leaf[x < m ? x : rot_a[x]] = need_leaf[x < m ? x : rot_b[x]] = 1;
  for (int j = 0; j < m; ++j)
    if (need_leaf[j]) f += fmt("  const gar_io l%d = gar_ldio(tin[%d] + e);\n", j, j);
  // operand text; values at placements >= m arrive from the other half once
  std::vector<char> got(nv, 0);
  auto fetch = [&](int x) {
    if (plc(x) < m || got[x]) return;
    got[x] = 1;
    const int vb = rot_b[x], va = rot_a[x];
    if (x < P)
      f += fmt("  const gar_io y%d = gar_xio(hb ? l%d : l%d);\n", x, vb, va);
    else
      f += fmt("  const gar_acc x%d = gar_xacc(hb ? v%d : v%d);\n", x, vb, va);
  };
  auto leaf = [&](int x) { return x < m ? fmt("l%d", x) : fmt("y%d", x); };
  auto opnd = [&](int x) {
    if (x < P) return "gar_wide(" + leaf(x) + ")";
    return plc(x) < m ? fmt("v%d", x) : fmt("x%d", x);
  };
  for (int L = 1; L <= maxlvl; ++L) {
    for (int k : comb[L]) {
      if (is_hi[k]) continue;
      const int v = P + k, a = fp.a[k], b = fp.b[k];
      fetch(a);
      fetch(b);
      if (mate[k] >= 0) {
        const int k2 = mate[k], v2 = P + k2;
        fetch(fp.a[k2]);
        fetch(fp.b[k2]);
        f += fmt("  const float2 w%d = __fadd2_rn(make_float2(", v) + opnd(a) + ", " + opnd(fp.a[k2]) +
             "), make_float2(" + opnd(b) + ", " + opnd(fp.b[k2]) + "));\n";
        f += fmt("  const gar_acc v%d = w%d.x, v%d = w%d.y;\n", v, v, v2, v);
      } else if (bf16_sum && (a < P || b < P)) {
        const int lf = a < P ? a : b, other = a < P ? b : a;
        f += fmt("  const gar_acc v%d = gar_addbf(", v) + leaf(lf) + ", " + opnd(other) + ");\n";
      } else {
        f += fmt("  const gar_acc v%d = gar_op(", v) + opnd(a) + ", " + opnd(b) + ");\n";
      }
    }
  }
  for (int p = 0; p < m; ++p) {
    const int v = fp.out[fp.origin[p]];
    const std::string st = fmt("gar_stio(tout[%d] + e, ", p) + opnd(v) + ");";
    f += (odd && p == m - 1) ? "  if (ok && !hb) " + st + "\n" : "  if (ok) " + st + "\n";
  }
  f += "}\n";
  s += f;

  s += fmt("extern \"C\" __global__ void __launch_bounds__(%d, %d) ", cg.threads, minb) + cg.kernel_name +
       "(const __grid_constant__ gar_args a) {\n";
  s += fmt("  __shared__ const gar_io *s_in[%d];\n  __shared__ gar_io *s_out[%d];\n", 2 * P, 2 * P);
  s += fmt("  for (int i = threadIdx.x; i < %d; i += blockDim.x) { s_in[i] = a.in[i]; s_out[i] = a.out[i]; }\n", 2 * P);
  s += "  __syncthreads();\n";
  // launched with programmatic stream serialisation: nothing is read before every
  // earlier kernel on the stream has completed
  s += "  asm volatile(\"griddepcontrol.wait;\" ::: \"memory\");\n";
  s += "  const int lane = threadIdx.x & 31, hb = lane >> 4;\n";
  s += fmt("  const gar_io *const *tin = s_in + (hb ? %d : 0);\n", m);
  s += fmt("  gar_io *const *tout = s_out + (hb ? %d : 0);\n", m);
  s += "  const gar_u64 npos = a.e_hi - a.e_lo;\n";
  s += "  const gar_u64 gw = ((gar_u64)blockIdx.x * blockDim.x + threadIdx.x) >> 5;\n";
  s += "  const gar_u64 nw = ((gar_u64)gridDim.x * blockDim.x) >> 5;\n";
  // 16 element positions per warp; a ragged last group reads the last position again
  // and stores nothing for the missing ones (every lane takes part in the shuffles)
  s += "  for (gar_u64 base = gw * 16; base < npos; base += nw * 16) {\n";
  s += "    const gar_u64 i = base + (gar_u64)(lane & 15);\n";
  s += "    const bool ok = i < npos;\n";
  s += "    gar_eval_sp(tin, tout, a.e_lo + (ok ? i : npos - 1), hb, ok);\n";
  s += "  }\n";
  s += "  asm volatile(\"griddepcontrol.launch_dependents;\" ::: \"memory\");\n}\n";
  cg.source = s;
  return cg;
}


CodegenResult generate_batched_source(const std::vector<const gar_plan *> &plans) {
  const gar_plan &p0 = *plans[0];
  int peak = 1;
  std::vector<Schedule> scs;
  for (const gar_plan *pl : plans) {
    scs.push_back(order_program(pl->prog));
    peak = std::max(peak, scs.back().peak_live);
  }
  // a row of n elements must split into whole vectors for every row to stay aligned
  int W = choose_width(p0.dtype, peak, 16);
  while (W > 1 && p0.n % W != 0) W /= 2;
  CodegenResult cg;
  cg.width = W;
  std::string name = "gar_batched_";
  for (const gar_plan *pl : plans)
    name += fmt("P%dS%d", pl->P, pl->S) + (pl->group == GAR_GROUP_XOR ? "x_" : "_");
  cg.kernel_name = name + dtype_tag(p0.dtype) + "_" + op_tag(p0.op) + fmt("_W%d", W);
  std::string s;
  s += fmt("#define GAR_DTYPE %d\n#define GAR_OP %d\n", p0.dtype, p0.op);
  s += fmt("#define GAR_FADD2 %d\n", tune_int("GAR_TUNE_FADD2", 0) != 0 ? 1 : 0);
  s += "#define GAR_LDH \"" + tune_str("GAR_TUNE_LDH", ".cs") + "\"\n";
  s += "#define GAR_STH \"" + tune_str("GAR_TUNE_STH", ".cs") + "\"\n";
  s += kSkeleton;
  s += fmt("#define GAR_W %d\n#define GAR_N %lluULL\n", W, (unsigned long long)p0.n);
  s += "struct gar_desc { int plan; int reserved; const void *in; void *out; };\n";
  s += "struct gar_bargs { const gar_desc *desc; gar_u64 count; };\n";
  // rows: input row r = in + r * n, output row r = out + r * n.  The generated eval
  // loads through RIN and stores through ROUT.
  for (size_t k = 0; k < plans.size(); ++k) {
    const gar_plan &pl = *plans[k];
    const bool rotate = pl.K != pl.P;
    std::string tag = fmt("p%zu", k);
    s += emit_block_of("gar_block_of_" + tag, pl.P, pl.n);
    auto ld = [](const std::string &r) { return "(in + GAR_N * (gar_u64)(" + r + "))"; };
    auto st = [](const std::string &r) { return "(out + GAR_N * (gar_u64)(" + r + "))"; };
    s += emit_eval(pl.prog, scs[k], tag, "const gar_io *in, gar_io *out", ld, st, rotate,
                   pl.group == GAR_GROUP_XOR);
  }
  s += "extern \"C\" __global__ void __launch_bounds__(256) " + cg.kernel_name +
       "(const __grid_constant__ gar_bargs a) {\n";
  s += "  const gar_u64 nvec = GAR_N / GAR_W;\n";
  s += "  const gar_u64 per = nvec + (GAR_N - nvec * GAR_W);\n";
  s += "  const gar_u64 total = a.count * per;\n";
  s += "  const gar_u64 stride = (gar_u64)gridDim.x * blockDim.x;\n";
  // A thread's next descriptor is loaded before its current item's contributions, so
  // with fewer threads than items the descriptor latency overlaps the data loads.
  s += "  gar_u64 g = (gar_u64)blockIdx.x * blockDim.x + threadIdx.x;\n";
  s += "  if (g >= total) return;\n";
  // launched with programmatic stream serialisation: nothing is read before every
  // earlier kernel on the stream has completed
  s += "  asm volatile(\"griddepcontrol.wait;\" ::: \"memory\");\n";
  s += "  gar_desc dn = a.desc[g / per];\n";
  s += "  for (; g < total; g += stride) {\n";
  s += "    const gar_u64 i = g / per, v = g - i * per;\n";
  s += "    const gar_desc d = dn;\n";
  s += "    if (g + stride < total) dn = a.desc[(g + stride) / per];\n";
  s += "    const gar_io *in = (const gar_io *)d.in;\n";
  s += "    gar_io *out = (gar_io *)d.out;\n";
  s += "    const bool aligned = (((gar_u64)in | (gar_u64)out) & (GAR_W * sizeof(gar_io) - 1)) == 0;\n";
  s += "    switch (d.plan) {\n";
  for (size_t k = 0; k < plans.size(); ++k) {
    const gar_plan &pl = *plans[k];
    const bool rotate = pl.K != pl.P;
    std::string tag = fmt("p%zu", k);
    std::string bo = "gar_block_of_" + tag;
    s += fmt("    case %zu:\n", k);
    s += "      if (v < nvec) {\n";
    s += "        const gar_u64 e0 = v * GAR_W;\n";
    if (rotate) {
      s += "        const int b0 = " + bo + "(e0);\n";
      s += "        if (aligned && (GAR_W == 1 || b0 == " + bo + "(e0 + GAR_W - 1))) gar_eval_" + tag +
           "<GAR_W>(in, out, e0, b0);\n";
      s += "        else for (int w = 0; w < GAR_W; ++w) gar_eval_" + tag + "<1>(in, out, e0 + w, " + bo +
           "(e0 + w));\n";
    } else {
      s += "        if (aligned) gar_eval_" + tag + "<GAR_W>(in, out, e0, 0);\n";
      s += "        else for (int w = 0; w < GAR_W; ++w) gar_eval_" + tag + "<1>(in, out, e0 + w, 0);\n";
    }
    s += "      } else {\n";
    s += "        const gar_u64 e = nvec * GAR_W + (v - nvec);\n";
    s += rotate ? "        gar_eval_" + tag + "<1>(in, out, e, " + bo + "(e));\n"
                : "        gar_eval_" + tag + "<1>(in, out, e, 0);\n";
    s += "      }\n      break;\n";
  }
  s += "    default: break;\n    }\n  }\n";
  s += "  asm volatile(\"griddepcontrol.launch_dependents;\" ::: \"memory\");\n}\n";
  cg.source = s;
  return cg;
}

}  // namespace gar
