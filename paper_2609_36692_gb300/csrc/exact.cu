// NormPre-L with exact eigenspace extraction (Sec. 3.2, App. B): the
// interaction matrix Gamma = Psi_a Psi_a^T (m_a x m_a, active orientation),
// its full symmetric eigendecomposition, and the selected set C = the up to r
// largest eigenvalues above one (Sec. 2.3).  The selected eigenpairs take the
// place of the sketch's Ritz pairs: Q = U_C (zero-padded to l = min(m_a, r)
// columns), K = diag(lambda_C^{-1/2} - 1), so the shared tail of the NormPre-L
// step (B^T = Psi_a^T Q, Q K, T = Psi + Q K B^T with the RMS-matched update)
// is unchanged, and ||T||_F^2 = m' - sum_C (lambda - 1) holds exactly.
//
// The same spectrum gives the spectral transformation energies of App. E:
// e_i = (sqrt(lambda_i) - 1)^2 summed over C (E_top), over lambda_i > 1 not in
// C (E_remain) and over 0 < lambda_i < 1 (E_sub); "nonzero" is read as
// lambda_i > 1e-6 lambda_max.
//
// Gamma is formed by k_gamma (fp32 FMA, 64 x 64 tiles); the dense symmetric
// eigensolver is cuSOLVER's syevd (fp32), loaded at run time with dlopen so
// that the rest of the library does not depend on it.  Matrices are taken one
// at a time per group (Gamma of one matrix is the workspace).
#include <cusolverDn.h>
#include <dlfcn.h>

#include <algorithm>
#include <mutex>
#include <string>

#include "common.cuh"
#include "internal.h"

namespace normpre {

namespace {

struct CusolverApi {
  bool ok = false;
  std::string why;
  cusolverStatus_t (*create)(cusolverDnHandle_t*) = nullptr;
  cusolverStatus_t (*destroy)(cusolverDnHandle_t) = nullptr;
  cusolverStatus_t (*set_stream)(cusolverDnHandle_t, cudaStream_t) = nullptr;
  cusolverStatus_t (*syevd_size)(cusolverDnHandle_t, cusolverEigMode_t, cublasFillMode_t, int, const float*, int,
                                 const float*, int*) = nullptr;
  cusolverStatus_t (*syevd)(cusolverDnHandle_t, cusolverEigMode_t, cublasFillMode_t, int, float*, int, float*,
                            float*, int, int*) = nullptr;
};

const CusolverApi& cusolver() {
  static CusolverApi api;
  static std::once_flag once;
  std::call_once(once, [] {
    void* lib = nullptr;
    for (const char* name : {"libcusolver.so.12", "libcusolver.so.11", "libcusolver.so"}) {
      lib = dlopen(name, RTLD_NOW | RTLD_LOCAL);
      if (lib) break;
    }
    if (!lib) {
      api.why = "libcusolver could not be loaded";
      return;
    }
    api.create = reinterpret_cast<decltype(api.create)>(dlsym(lib, "cusolverDnCreate"));
    api.destroy = reinterpret_cast<decltype(api.destroy)>(dlsym(lib, "cusolverDnDestroy"));
    api.set_stream = reinterpret_cast<decltype(api.set_stream)>(dlsym(lib, "cusolverDnSetStream"));
    api.syevd_size = reinterpret_cast<decltype(api.syevd_size)>(dlsym(lib, "cusolverDnSsyevd_bufferSize"));
    api.syevd = reinterpret_cast<decltype(api.syevd)>(dlsym(lib, "cusolverDnSsyevd"));
    api.ok = api.create && api.destroy && api.set_stream && api.syevd_size && api.syevd;
    if (!api.ok) api.why = "libcusolver lacks the syevd entry points";
  });
  return api;
}

// Gamma[i][j] = sum_k A[i][k] A[j][k] over the active rows A of Psi (row-major,
// row stride ld): rows of Psi (TRANS = false) or its columns (TRANS = true).
// Gamma[i][j] and Gamma[j][i] take the same products in the same order, so
// the result is exactly symmetric.
struct GammaArgs {
  const float* psi;
  int64_t ld;
  int64_t m, k;         // m_a, n_a
  float* gamma;         // [m][m]
};
template <bool TRANS>
__global__ void __launch_bounds__(256) k_gamma(const __grid_constant__ GammaArgs a) {
  __shared__ float As[16][64 + 4], Bs[16][64 + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int64_t i0 = static_cast<int64_t>(blockIdx.y) * 64, j0 = static_cast<int64_t>(blockIdx.x) * 64;
  float acc[4][4] = {};
  for (int64_t k0 = 0; k0 < a.k; k0 += 16) {
    for (int e = threadIdx.x; e < 16 * 64; e += 256) {
      // consecutive threads read consecutive addresses: K for rows of Psi,
      // the element index for its columns
      const int ii = TRANS ? (e & 63) : (e >> 4), kk = TRANS ? (e >> 6) : (e & 15);
      const int64_t k = k0 + kk, i = i0 + ii, j = j0 + ii;
      As[kk][ii] = (i < a.m && k < a.k) ? (TRANS ? a.psi[k * a.ld + i] : a.psi[i * a.ld + k]) : 0.f;
      Bs[kk][ii] = (j < a.m && k < a.k) ? (TRANS ? a.psi[k * a.ld + j] : a.psi[j * a.ld + k]) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float av[4], bv[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) av[r] = As[kk][ty * 4 + r];
#pragma unroll
      for (int c = 0; c < 4; ++c) bv[c] = Bs[kk][tx * 4 + c];
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(av[r], bv[c], acc[r][c]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int64_t i = i0 + ty * 4 + r;
    if (i >= a.m) continue;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int64_t j = j0 + tx * 4 + c;
      if (j < a.m) a.gamma[i * a.m + j] = acc[r][c];
    }
  }
}

// From the ascending eigenvalues w and the eigenvectors (column j of the
// column-major n x n result = eigenvector of w[j]) of one matrix: all
// eigenvalues descending, Q = the l leading eigenvectors, Ritz values, Z = I,
// K = diag(lambda^{-1/2} - 1) on C, the step statistics and the energies.
struct SelectArgs {
  const float* w;            // [n] ascending
  const float* vec;          // [n][n], column j at vec + j n
  const int* info;           // syevd status
  int64_t n, n_a;
  int l, rank, k_orient;
  float* eig_all;            // [n] descending
  float* q;                  // [n][l]
  float* ritz;               // [l]
  float* z;                  // [l][l]
  float* kmat;               // [l][l]
  float* stats;              // [8]
  double* diag;              // [8] or null: E_top, E_remain, E_sub, E_global
  const int* count;
  int mat_id;
  int* flags;
};
__global__ void __launch_bounds__(256) k_exact_select(const __grid_constant__ SelectArgs a) {
  const int64_t n = a.n;
  const int l = a.l;
  for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < n * l;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t i = e / l;
    const int c = static_cast<int>(e - i * l);
    a.q[e] = a.vec[(n - 1 - c) * n + i];
  }
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    a.eig_all[i] = a.w[n - 1 - i];
  if (blockIdx.x != 0) return;
  __shared__ double red[32];
  __shared__ int nc_s;
  const int rr = min(a.rank, l);
  if (threadIdx.x == 0) {
    int nc = 0;
    for (int c = 0; c < rr; ++c) {
      if (!(a.w[n - 1 - c] > 1.f)) break;   // descending: the first lambda <= 1 ends C
      ++nc;
    }
    nc_s = nc;
  }
  __syncthreads();
  const int nc = nc_s;
  for (int e = threadIdx.x; e < l * l; e += blockDim.x) {
    const int r = e / l, c = e % l;
    a.z[e] = (r == c) ? 1.f : 0.f;
    a.kmat[e] = (r == c && c < nc) ? rsqrtf(a.w[n - 1 - c]) - 1.f : 0.f;
  }
  for (int c = threadIdx.x; c < l; c += blockDim.x) a.ritz[c] = a.w[n - 1 - c];
  // sums over the spectrum in fp64: the excess of C, and the three energies
  const double lmax = a.w[n - 1];
  const double floor_ = 1e-6 * lmax;
  double ex = 0, top = 0, rem = 0, sub = 0;
  for (int64_t i = threadIdx.x; i < n; i += blockDim.x) {
    const int64_t c = n - 1 - i;               // rank in descending order
    const double lam = a.w[i];
    const double e = (sqrt(fmax(lam, 0.0)) - 1.0) * (sqrt(fmax(lam, 0.0)) - 1.0);
    if (c < nc) {
      ex += lam - 1.0;
      top += e;
    } else if (lam > 1.0) {
      rem += e;
    } else if (lam > floor_ && lam < 1.0) {
      sub += e;
    }
  }
  ex = block_sum(ex, red);
  top = block_sum(top, red);
  rem = block_sum(rem, red);
  sub = block_sum(sub, red);
  if (threadIdx.x == 0) {
    const float mprime = static_cast<float>(a.count[a.mat_id]);
    a.stats[0] = static_cast<float>(a.k_orient);
    a.stats[1] = mprime;
    a.stats[2] = fmaxf(mprime - static_cast<float>(ex), 0.f);
    a.stats[3] = static_cast<float>(nc);
    a.stats[4] = static_cast<float>(l);
    a.stats[5] = static_cast<float>(a.n_a);
    a.stats[6] = static_cast<float>(n);
    a.stats[7] = 0.f;
    if (a.diag) {
      a.diag[0] = top;
      a.diag[1] = rem;
      a.diag[2] = sub;
      a.diag[3] = top + rem + sub;
    }
    if (*a.info != 0) raise_flag(a.flags, kFlagNumeric);
    if (!isfinite(lmax)) raise_flag(a.flags, kFlagNonfinite);
  }
}

}  // namespace

int exact_available(std::string* why) {
  const CusolverApi& api = cusolver();
  if (!api.ok && why) *why = api.why;
  return api.ok ? 1 : 0;
}

cudaError_t exact_group_alloc(SketchGroup& g, std::vector<void*>& allocs, std::string* why) {
  const CusolverApi& api = cusolver();
  if (!api.ok) {
    if (why) *why = api.why;
    return cudaErrorNotSupported;
  }
  const int64_t big = std::max(g.rows, g.cols);
  auto alloc = [&](void** p, size_t bytes) -> cudaError_t {
    cudaError_t e = cudaMalloc(p, bytes);
    if (e == cudaSuccess) allocs.push_back(*p);
    return e;
  };
  cudaError_t e;
  if ((e = alloc(reinterpret_cast<void**>(&g.gamma), sizeof(float) * big * big))) return e;
  if ((e = alloc(reinterpret_cast<void**>(&g.eig_w), sizeof(float) * big))) return e;
  if ((e = alloc(reinterpret_cast<void**>(&g.eig_all), sizeof(float) * big * g.batch))) return e;
  if ((e = alloc(reinterpret_cast<void**>(&g.eig_info), sizeof(int)))) return e;
  cusolverDnHandle_t h = nullptr;
  if (api.create(&h) != CUSOLVER_STATUS_SUCCESS) {
    if (why) *why = "cusolverDnCreate failed";
    return cudaErrorNotSupported;
  }
  g.solver = h;
  int lwork = 0;
  for (int64_t n : {g.rows, g.cols}) {
    int lw = 0;
    if (api.syevd_size(h, CUSOLVER_EIG_MODE_VECTOR, CUBLAS_FILL_MODE_LOWER, static_cast<int>(n), g.gamma,
                       static_cast<int>(n), g.eig_w, &lw) != CUSOLVER_STATUS_SUCCESS) {
      if (why) *why = "cusolverDnSsyevd_bufferSize failed";
      return cudaErrorNotSupported;
    }
    lwork = std::max(lwork, lw);
  }
  g.eig_lwork = lwork;
  return alloc(reinterpret_cast<void**>(&g.eig_work), sizeof(float) * std::max(lwork, 1));
}

void exact_group_free(SketchGroup& g) {
  if (g.solver) {
    cusolver().destroy(static_cast<cusolverDnHandle_t>(g.solver));
    g.solver = nullptr;
  }
}

cudaError_t exact_eigs(SketchGroup& g, const SketchParams& p, int l, const int* mat_ids_host, const int* count,
                       double* diag, int* flags, cudaStream_t s, ProfileHook* prof) {
  ProfileHook none;
  if (!prof) prof = &none;
  const CusolverApi& api = cusolver();
  if (!api.ok || !g.solver) return cudaErrorNotSupported;
  const bool rows_active = (p.k == 0);
  const int64_t m_a = rows_active ? g.rows : g.cols, n_a = rows_active ? g.cols : g.rows;
  const int64_t big = std::max(g.rows, g.cols);
  const int64_t vbs = big * g.lmax;
  const int64_t sq = static_cast<int64_t>(g.lmax) * g.lmax;
  cusolverDnHandle_t h = static_cast<cusolverDnHandle_t>(g.solver);
  if (api.set_stream(h, s) != CUSOLVER_STATUS_SUCCESS) return cudaErrorUnknown;
  for (int b = 0; b < g.batch; ++b) {
    GammaArgs ga;
    ga.psi = g.psi + b * g.rows * g.ld;
    ga.ld = g.ld;
    ga.m = m_a;
    ga.k = n_a;
    ga.gamma = g.gamma;
    const dim3 grid(static_cast<unsigned>(cdiv(m_a, 64)), static_cast<unsigned>(cdiv(m_a, 64)));
    prof->begin(kProfGamma, s);
    if (rows_active) k_gamma<false><<<grid, 256, 0, s>>>(ga);
    else k_gamma<true><<<grid, 256, 0, s>>>(ga);
    cudaError_t e = cudaGetLastError();
    if (e) return e;
    prof->end(kProfGamma, s, 1);
    prof->begin(kProfSyevd, s);
    if (api.syevd(h, CUSOLVER_EIG_MODE_VECTOR, CUBLAS_FILL_MODE_LOWER, static_cast<int>(m_a), g.gamma,
                  static_cast<int>(m_a), g.eig_w, g.eig_work, g.eig_lwork, g.eig_info) != CUSOLVER_STATUS_SUCCESS)
      return cudaErrorUnknown;
    SelectArgs sa;
    sa.w = g.eig_w;
    sa.vec = g.gamma;
    sa.info = g.eig_info;
    sa.n = m_a;
    sa.n_a = n_a;
    sa.l = l;
    sa.rank = p.rank;
    sa.k_orient = p.k;
    sa.eig_all = g.eig_all + b * big;
    sa.q = g.q + b * vbs;
    sa.ritz = g.ritz + static_cast<int64_t>(b) * g.lmax;
    sa.z = g.zvec + b * sq;
    sa.kmat = g.kmat + b * sq;
    sa.stats = g.stats + b * 8;
    sa.diag = diag ? diag + 8 * static_cast<int64_t>(mat_ids_host[b]) : nullptr;
    sa.count = count;
    sa.mat_id = mat_ids_host[b];
    sa.flags = flags;
    const int blocks = static_cast<int>(std::min<int64_t>(cdiv(m_a * l, 256), 1024));
    k_exact_select<<<std::max(blocks, 1), 256, 0, s>>>(sa);
    if ((e = cudaGetLastError())) return e;
    prof->end(kProfSyevd, s, 1);
  }
  return cudaSuccess;
}

}  // namespace normpre
