// Allocation-free variant of the column-active momentum + relaxed tangent +
// diagonal-Gram normalization (the kernels of normalize.cu).
//
// Some callers cannot call cudaMalloc at the time they need this step: code
// running inside a memory pool or allocator callback, a framework whose
// allocator must not be re-entered, or a process whose device memory is fully
// reserved up front.  For them this entry point takes its scratch (the
// per-row-block column sums and the per-column coefficients) from a fixed
// array in the library's own device memory instead of the handle's
// workspace.  It performs no allocation or free of any kind.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds it (kNoAllocScratchBytes) until the process exits, and every
// call shares it.  Host code only sees a stand-in for it, so its device
// address is fetched with cudaGetSymbolAddress once per device, on the first
// call made with that device current.
#include <cuda_runtime.h>

#include <mutex>
#include <string>

#include "../../include/normpre.h"
#include "internal.h"

namespace normpre {

constexpr size_t kNoAllocScratchBytes = size_t(8) << 20;   // 8 MiB
constexpr int kNoAllocMaxDevices = 64;

// [0, 16): count of nonzero columns and the status word; then the column
// partial sums and coefficients used by launch_normalize_cols.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

namespace {
std::mutex g_noalloc_mutex;
void* g_noalloc_addr[kNoAllocMaxDevices] = {};

// Failures are reported through normpre_last_error(NULL), like every other
// call without a handle.
int noalloc_fail(int code, const std::string& msg) {
  set_thread_error(msg);
  return code;
}
}  // namespace

}  // namespace normpre

using namespace normpre;

extern "C" int normpre_normalize_cols_noalloc(int64_t rows, int64_t cols, float mu, const void* G,
                                              int g_dtype, float* M, const void* W, int w_dtype,
                                              float* Psi, void* stream) {
  if (!G || !M || !W || !Psi) return noalloc_fail(NORMPRE_ERR_ARG, "null tensor pointer");
  if (rows < 1 || cols < 1 || rows > 65536 || cols > 65536)
    return noalloc_fail(NORMPRE_ERR_SHAPE, "each dimension must be in [1, 65536]");
  if ((g_dtype != NORMPRE_F32 && g_dtype != NORMPRE_BF16) || (w_dtype != NORMPRE_F32 && w_dtype != NORMPRE_BF16))
    return noalloc_fail(NORMPRE_ERR_DTYPE, "dtype must be NORMPRE_F32 or NORMPRE_BF16");
  auto aligned16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  if (!aligned16(G) || !aligned16(M) || !aligned16(W) || !aligned16(Psi))
    return noalloc_fail(NORMPRE_ERR_ALIGN, "tensors must be 16-byte aligned");
  const size_t need = 256 + normalize_cols_scratch_bytes(rows, cols, 1);
  if (need > kNoAllocScratchBytes)
    return noalloc_fail(NORMPRE_ERR_SHAPE,
                        "rows x cols needs " + std::to_string(need) + " bytes of scratch; the fixed "
                        "array holds " + std::to_string(kNoAllocScratchBytes) +
                        " (at most about 87 million elements)");
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return noalloc_fail(NORMPRE_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev < 0 || dev >= kNoAllocMaxDevices) return noalloc_fail(NORMPRE_ERR_ARG, "device index out of range");
  void* base = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (!g_noalloc_addr[dev]) {
      e = cudaGetSymbolAddress(&g_noalloc_addr[dev], g_noalloc_scratch);
      if (e != cudaSuccess) {
        g_noalloc_addr[dev] = nullptr;
        return noalloc_fail(NORMPRE_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
      }
    }
    base = g_noalloc_addr[dev];
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* p = static_cast<char*>(base);
  int* count = reinterpret_cast<int*>(p);
  int* flags = reinterpret_cast<int*>(p + 4);
  // the previous call's counter and status word must not leak into this one
  e = cudaMemsetAsync(p, 0, 16, s);
  if (e != cudaSuccess) return noalloc_fail(NORMPRE_ERR_CUDA, std::string("cudaMemsetAsync: ") + cudaGetErrorString(e));
  NormLaunch a;
  a.n = 1;
  a.rows = rows;
  a.cols = cols;
  a.g_dtype = g_dtype;
  a.w_dtype = w_dtype;
  a.psi_dtype = 0;
  a.G[0] = G;
  a.M[0] = M;
  a.W[0] = W;
  a.psi[0] = Psi;
  a.mat_id[0] = 0;
  a.psi_ld = cols;
  a.mu = mu;
  a.count = count;
  a.flags = flags;
  a.col_part = reinterpret_cast<double*>(p + 256);
  a.col_coef = reinterpret_cast<float2*>(p + 256 + normalize_cols_part_bytes(rows, cols, 1));
  e = launch_normalize_cols(a, s);
  if (e != cudaSuccess) return noalloc_fail(NORMPRE_ERR_CUDA, std::string("launch: ") + cudaGetErrorString(e));
  return NORMPRE_OK;
}
