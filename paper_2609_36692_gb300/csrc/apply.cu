// NormPre-G weight update (Algorithm 1, consistent update RMS of Sec. 3.1):
//   W <- W - lr (target * O_k^{-1}(T) / RMS(T) + wd W),  RMS(T) = ||T||_F / sqrt(mn).
// T is the Newton-Schulz result, already in the stored layout (the iteration
// commutes with transposition), so O_k^{-1} is free.  ||T||_F^2 arrives as
// per-tile partial sums written by the last Newton-Schulz epilogue; every CTA
// folds the partials of its matrix in the same fixed order.
#include <type_traits>

#include "common.cuh"
#include "internal.h"

namespace normpre {

template <typename TW, typename TT, bool VEC>
__global__ void __launch_bounds__(256) k_apply_g(const __grid_constant__ ApplyLaunch a) {
  __shared__ double red[32];
  __shared__ float scale_s;
  const int b = blockIdx.y;
  double s = 0;
  for (int i = threadIdx.x; i < a.n_part; i += blockDim.x) s += a.sq_part[b][i];
  s = block_sum(s, red);
  if (threadIdx.x == 0) {
    // formed by one thread: fp64 throughput is low on this part
    const double mn = static_cast<double>(a.rows) * static_cast<double>(a.cols);
    scale_s = s > 0 ? static_cast<float>(a.target * sqrt(mn / s)) : 0.f;
    if (blockIdx.x == 0 && a.stats[b]) {
      a.stats[b][0] = static_cast<float>(a.k);
      a.stats[b][1] = a.count ? static_cast<float>(a.count[a.mat_id[b]]) : 0.f;
      a.stats[b][2] = static_cast<float>(s);
    }
  }
  __syncthreads();
  const float cw = 1.f - a.lr * a.wd, ct = -a.lr * scale_s;
  TW* W = static_cast<TW*>(a.W[b]);
  const TT* T = static_cast<const TT*>(a.T[b]);
  if (VEC) {
    const uint32_t cpr = static_cast<uint32_t>(a.cols / 8);
    const uint32_t nvec = static_cast<uint32_t>(a.rows) * cpr;
    for (uint32_t v = blockIdx.x * blockDim.x + threadIdx.x; v < nvec; v += gridDim.x * blockDim.x) {
      const uint32_t r = v / cpr, c = (v - r * cpr) * 8;
      float w[8], t[8];
      load8(W + static_cast<int64_t>(r) * a.cols + c, w);
      load8(T + static_cast<int64_t>(r) * a.t_ld + c, t);
#pragma unroll
      for (int e = 0; e < 8; ++e) w[e] = fmaf(cw, w[e], ct * t[e]);
      store8(W + static_cast<int64_t>(r) * a.cols + c, w);
    }
  } else {
    const int64_t n = a.rows * a.cols;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
      const int64_t r = i / a.cols, c = i - r * a.cols;
      const float w = to_f32(W[i]);
      W[i] = from_f32<TW>(fmaf(cw, w, ct * to_f32(T[r * a.t_ld + c])));
    }
  }
}

cudaError_t launch_apply_g(const ApplyLaunch& a, cudaStream_t s) {
  if (a.n <= 0) return cudaSuccess;
  const bool vec = (a.cols % 8 == 0) && (a.t_ld % 8 == 0) &&
                   static_cast<uint64_t>(a.rows) * static_cast<uint64_t>(a.cols) / 8 < (1ull << 31);
  const int64_t work = vec ? a.rows * a.cols / 8 : a.rows * a.cols;
  int64_t per = cdiv(work, 256);
  const int64_t cap = cdiv(static_cast<int64_t>(device_sm_count()) * 8, a.n);
  if (per > cap) per = cap;
  if (per < 1) per = 1;
  const dim3 grid(static_cast<unsigned>(per), static_cast<unsigned>(a.n));
  auto go = [&](auto* tw, auto* tt) {
    using TW = std::remove_pointer_t<decltype(tw)>;
    using TT = std::remove_pointer_t<decltype(tt)>;
    if (vec) k_apply_g<TW, TT, true><<<grid, 256, 0, s>>>(a);
    else k_apply_g<TW, TT, false><<<grid, 256, 0, s>>>(a);
    return cudaGetLastError();
  };
  if (a.w_dtype == 0 && a.t_dtype == 0) return go((float*)0, (float*)0);
  if (a.w_dtype == 0 && a.t_dtype == 1) return go((float*)0, (bf16*)0);
  if (a.w_dtype == 1 && a.t_dtype == 0) return go((bf16*)0, (float*)0);
  return go((bf16*)0, (bf16*)0);
}

// Descent-alignment sums of a Newton-Schulz step: <G, T>, ||G||^2, ||T||^2 of
// every matrix, T in the stored layout (row stride t_ld), accumulated into
// diag[4..6] with fp64 atomics (diagnostics: not bitwise reproducible).
__global__ void __launch_bounds__(256) k_diag_gt(const __grid_constant__ DiagLaunch a) {
  __shared__ double red[32];
  const int b = blockIdx.y;
  double gt = 0, gg = 0, tt = 0;
  const int64_t n = a.rows * a.cols;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t r = i / a.cols, c = i - r * a.cols;
    const float g = a.g_dtype ? to_f32(static_cast<const bf16*>(a.G[b])[i]) : static_cast<const float*>(a.G[b])[i];
    const float t = a.t_dtype ? to_f32(static_cast<const bf16*>(a.T[b])[r * a.t_ld + c])
                              : static_cast<const float*>(a.T[b])[r * a.t_ld + c];
    gt += static_cast<double>(g) * t;
    gg += static_cast<double>(g) * g;
    tt += static_cast<double>(t) * t;
  }
  gt = block_sum(gt, red);
  gg = block_sum(gg, red);
  tt = block_sum(tt, red);
  if (threadIdx.x == 0) {
    atomicAdd(a.diag[b] + 4, gt);
    atomicAdd(a.diag[b] + 5, gg);
    atomicAdd(a.diag[b] + 6, tt);
  }
}

cudaError_t launch_diag_gt(const DiagLaunch& a, cudaStream_t s) {
  if (a.n <= 0) return cudaSuccess;
  int64_t per = cdiv(a.rows * a.cols, 256 * 8);
  const int64_t cap = cdiv(static_cast<int64_t>(device_sm_count()) * 4, a.n);
  per = std::max<int64_t>(1, std::min(per, cap));
  k_diag_gt<<<dim3(static_cast<unsigned>(per), static_cast<unsigned>(a.n)), 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace normpre
