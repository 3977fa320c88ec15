// Muon baseline (the paper's comparison optimizer, Sec. 4 and App. A): the
// Newton-Schulz iteration of Muon (Sec. 2.1) applied to the momentum itself,
// with the same RMS-matched update as NormPre (Sec. 3.1).  It shares the
// Newton-Schulz plan and the update kernel with NormPre-G; what is specific
// to it is this elementwise pass: M_t = mu M_{t-1} + G_t, written back and
// copied into the Newton-Schulz input buffer, with fp64 partial sums of
// ||M_t||^2 per row block that a second kernel folds (fixed order) into the
// prescale 1 / (||M_t||_F + eps).
#include <type_traits>

#include "common.cuh"
#include "internal.h"

namespace normpre {

template <typename TG, typename TP, bool VEC>
__global__ void __launch_bounds__(256) k_momentum_copy(const __grid_constant__ NormLaunch a, double* part, int nblk,
                                                       int stride) {
  __shared__ double red[32];
  const int b = blockIdx.y, blk = blockIdx.x;
  const int64_t rows = a.rows, cols = a.cols;
  const int64_t rpb = (rows + nblk - 1) / nblk;
  const int64_t r0 = static_cast<int64_t>(blk) * rpb, r1 = min(rows, r0 + rpb);
  const TG* g = static_cast<const TG*>(a.G[b]);
  float* M = a.M[b];
  TP* psi = static_cast<TP*>(a.psi[b]);
  float ss = 0.f;
  if (r1 > r0) {
    if (VEC) {
      const int64_t cpr = cols / 8, total = (r1 - r0) * cpr;
      for (int64_t i = threadIdx.x; i < total; i += blockDim.x) {
        const int64_t r = r0 + i / cpr, c = (i % cpr) * 8;
        float gv[8], mv[8];
        load8(g + r * cols + c, gv);
        load8_cg(M + r * cols + c, mv);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          mv[e] = fmaf(a.mu, mv[e], gv[e]);
          ss = fmaf(mv[e], mv[e], ss);
        }
        store8(M + r * cols + c, mv);
        store8(psi + r * a.psi_ld + c, mv);
      }
    } else {
      const int64_t total = (r1 - r0) * cols;
      for (int64_t i = threadIdx.x; i < total; i += blockDim.x) {
        const int64_t r = r0 + i / cols, c = i % cols;
        const float m = fmaf(a.mu, M[r * cols + c], to_f32(g[r * cols + c]));
        M[r * cols + c] = m;
        psi[r * a.psi_ld + c] = from_f32<TP>(m);
        ss = fmaf(m, m, ss);
      }
    }
  }
  const double s = block_sum(static_cast<double>(ss), red);
  if (threadIdx.x == 0) {
    part[static_cast<int64_t>(b) * stride + blk] = s;
    if (!isfinite(s)) raise_flag(a.flags, kFlagNonfinite);
  }
}

__global__ void k_muon_prescale(const double* part, int nblk, int stride, int batch, float* inscale, float eps) {
  for (int b = threadIdx.x; b < batch; b += blockDim.x) {
    double s = 0.0;
    for (int i = 0; i < nblk; ++i) s += part[static_cast<int64_t>(b) * stride + i];
    inscale[b] = static_cast<float>(1.0 / (sqrt(s) + static_cast<double>(eps)));
  }
}

cudaError_t launch_momentum_copy(const NormLaunch& a, double* part, int nblk, int stride, cudaStream_t s) {
  if (a.n <= 0 || a.rows <= 0 || a.cols <= 0) return cudaSuccess;
  const bool vec = (a.cols % 8 == 0) && (a.psi_ld % 8 == 0);
  const dim3 grid(static_cast<unsigned>(nblk), static_cast<unsigned>(a.n));
  auto go = [&](auto* tg, auto* tp) {
    using TG = std::remove_pointer_t<decltype(tg)>;
    using TP = std::remove_pointer_t<decltype(tp)>;
    if (vec) k_momentum_copy<TG, TP, true><<<grid, 256, 0, s>>>(a, part, nblk, stride);
    else k_momentum_copy<TG, TP, false><<<grid, 256, 0, s>>>(a, part, nblk, stride);
    return cudaGetLastError();
  };
  if (a.g_dtype == 0 && a.psi_dtype == 0) return go((float*)0, (float*)0);
  if (a.g_dtype == 0 && a.psi_dtype == 1) return go((float*)0, (bf16*)0);
  if (a.g_dtype == 1 && a.psi_dtype == 0) return go((bf16*)0, (float*)0);
  return go((bf16*)0, (bf16*)0);
}

cudaError_t launch_muon_prescale(const double* part, int nblk, int stride, int batch, float* inscale, float eps,
                                 cudaStream_t s) {
  k_muon_prescale<<<1, 256, 0, s>>>(part, nblk, stride, batch, inscale, eps);
  return cudaGetLastError();
}

}  // namespace normpre
