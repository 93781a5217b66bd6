// Run-time compilation of the generated fused / batched kernels for sm_103a.
//
// Compilation (NVRTC, source -> CUBIN) needs no GPU; loading (cudaLibraryLoadData)
// does.  Compiled kernels are cached for the life of the process, keyed by their full
// source text, so plans with the same program share one kernel.
#include <cuda_runtime.h>
#include <nvrtc.h>

#include <memory>
#include <mutex>
#include <string>
#include <unordered_map>

#include "gar_internal.hpp"

namespace gar {
namespace {

std::mutex g_mu;
std::unordered_map<std::string, std::unique_ptr<JitKernel>> g_cache;

}  // namespace

int jit_compile(const CodegenResult &cg, JitKernel **out) {
  std::lock_guard<std::mutex> lock(g_mu);
  auto it = g_cache.find(cg.source);
  if (it != g_cache.end()) {
    *out = it->second.get();
    return GAR_OK;
  }
  nvrtcProgram prog;
  if (nvrtcCreateProgram(&prog, cg.source.c_str(), "gar_generated.cu", 0, nullptr, nullptr) !=
      NVRTC_SUCCESS) {
    set_error("nvrtcCreateProgram failed");
    return GAR_EJIT;
  }
  const char *opts[] = {"--gpu-architecture=sm_103a", "--std=c++17", "-lineinfo",
                        "--fmad=false", "--ftz=false", "--prec-div=true", "--prec-sqrt=true"};
  nvrtcResult rc = nvrtcCompileProgram(prog, (int)(sizeof opts / sizeof opts[0]), opts);
  if (rc != NVRTC_SUCCESS) {
    size_t n = 0;
    nvrtcGetProgramLogSize(prog, &n);
    std::string log(n, '\0');
    if (n) nvrtcGetProgramLog(prog, &log[0]);
    nvrtcDestroyProgram(&prog);
    set_error("NVRTC compile of " + cg.kernel_name + " failed: " + log);
    return GAR_EJIT;
  }
  size_t bytes = 0;
  if (nvrtcGetCUBINSize(prog, &bytes) != NVRTC_SUCCESS || bytes == 0) {
    nvrtcDestroyProgram(&prog);
    set_error("NVRTC produced no CUBIN for " + cg.kernel_name);
    return GAR_EJIT;
  }
  auto k = std::make_unique<JitKernel>();
  k->cubin.resize(bytes);
  nvrtcGetCUBIN(prog, k->cubin.data());
  nvrtcDestroyProgram(&prog);
  k->name = cg.kernel_name;
  k->source = cg.source;
  k->width = cg.width;
  k->table_copies = cg.table_copies;
  k->threads = cg.threads;
  k->form = cg.form;
  *out = k.get();
  g_cache.emplace(cg.source, std::move(k));
  return GAR_OK;
}

int jit_load(JitKernel *k) {
  std::lock_guard<std::mutex> lock(g_mu);
  if (k->loaded) return GAR_OK;
  cudaLibrary_t lib = nullptr;
  cudaError_t e = cudaLibraryLoadData(&lib, k->cubin.data(), nullptr, nullptr, 0, nullptr,
                                      nullptr, 0);
  if (e != cudaSuccess) return cuda_fail(e, "cudaLibraryLoadData");
  cudaKernel_t kern = nullptr;
  e = cudaLibraryGetKernel(&kern, lib, k->name.c_str());
  if (e != cudaSuccess) {
    cudaLibraryUnload(lib);
    return cuda_fail(e, "cudaLibraryGetKernel");
  }
  int nb = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, (const void *)kern, k->threads, 0);
  if (e != cudaSuccess || nb <= 0) {
    cudaGetLastError();
    nb = 1;
  }
  cudaFuncAttributes fa{};
  if (cudaFuncGetAttributes(&fa, (const void *)kern) == cudaSuccess) {
    k->regs = fa.numRegs;
    k->local_bytes = (int)fa.localSizeBytes;
  } else {
    cudaGetLastError();
  }
  k->library = lib;
  k->kernel = (void *)kern;
  k->blocks_per_sm = nb;
  k->loaded = true;
  return GAR_OK;
}

}  // namespace gar
