// Fused momentum + relaxed tangent momentum + diagonal-Gram normalization
// (Algorithm 1 of the paper: M_t = mu M_{t-1} + G_t; x_i = m_i - <m_i, w_i> w_i
// for every active row; Psi = D(X)^{-1} X, Eq. 3).
//
// Row-active steps (k = 0): one CTA per stored row; the row of M and W stays in
// registers between the two block reductions (<m, w>, then ||x||^2), so the
// step reads G, M_{t-1}, W once and writes M_t, Psi once, with 16-byte vector
// accesses.
//
// Column-active steps (k = 1): the reduction runs down the columns of the
// row-major layout.  Pass A streams G, M_{t-1}, W once, writes M_t and per-
// (row block, column) partial sums of ||m||^2, <m, w> and ||w||^2; a small
// pass folds the partials (in fp64, fixed order, no atomics on floats) into
// a_j = <m_j, w_j> and 1/||x_j|| with ||x||^2 = ||m||^2 - a^2 (2 - ||w||^2);
// pass B re-reads M_t and W and writes Psi.
//
// Zero active rows (undefined in Eq. 3) give zero rows of Psi; count[] gets
// the number of nonzero rows m' (so ||Psi||_F^2 = m').
//
// The tangent step subtracts c_i w_i with c_i = <m_i, w_i> (relaxed, the
// paper's), <m_i, w_i> / ||w_i||^2 (strict tangent ablation; 0 for a zero
// weight row) or 0 (no-tangent ablation), Table 5a.  The strict projection
// of a momentum row parallel to its weight row leaves only rounding, which
// would normalize to a unit row of noise: with the coefficient from fp32
// sums that residue is up to ~1e-5 of ||m_i||, so a strict-tangent row
// whose x_i is at most 1e-3 of ||m_i|| is taken as zero (the kernels'
// fp32 resolution of the projection).  Column-active strict steps sum
// ||x_j||^2 from the subtracted values in an extra pass (the closed form
// ||m||^2 - <m, w>^2 / ||w||^2 cancels for such columns).
#include <type_traits>

#include "common.cuh"
#include "internal.h"

namespace normpre {

constexpr int kColStatsRB = 256;  // rows per block of pass A (one partial sum per block and column)
constexpr int kColApplyRB = 64;   // rows per block of pass B
constexpr int kColThreads = 256;  // 32 column chunks of 8 x 8 row lanes

// c_i of the tangent step for mode 0 relaxed, 1 none, 2 strict (mw = <m_i, w_i>,
// ww = ||w_i||^2).
__device__ __forceinline__ float tangent_coef(int mode, float mw, float ww) {
  if (mode == 0) return mw;
  if (mode == 2) return ww > 0.f ? mw / ww : 0.f;
  return 0.f;
}

size_t normalize_cols_part_bytes(int64_t rows, int64_t cols, int n) {
  return static_cast<size_t>(n) * cdiv(rows, kColStatsRB) * cols * 3 * sizeof(double);
}

size_t normalize_cols_scratch_bytes(int64_t rows, int64_t cols, int n) {
  const int64_t nrb = cdiv(rows, kColStatsRB);
  return static_cast<size_t>(n) * nrb * cols * 3 * sizeof(double) +
         static_cast<size_t>(n) * cols * sizeof(float2) + 256;
}

// ---------------------------------------------------------------------------
// row-active, vector path (cols % 8 == 0, cols <= 16 * blockDim)
// ---------------------------------------------------------------------------
template <typename TG, typename TW, typename TP>
__global__ void __launch_bounds__(1024) k_norm_rows_vec(const __grid_constant__ NormLaunch a) {
  __shared__ float red[32];
  const int b = blockIdx.y;
  const int64_t row = blockIdx.x;
  const int64_t cols = a.cols;
  const TG* g = static_cast<const TG*>(a.G[b]) + row * cols;
  float* M = a.M[b] + row * cols;
  const TW* w = static_cast<const TW*>(a.W[b]) + row * cols;
  TP* psi = static_cast<TP*>(a.psi[b]) + row * a.psi_ld;
  float m[2][8], wv[2][8];
  float dot = 0.f, wsq = 0.f;
#pragma unroll
  for (int c = 0; c < 2; ++c) {
    const int64_t j = (static_cast<int64_t>(c) * blockDim.x + threadIdx.x) * 8;
    if (j < cols) {
      float gv[8], mp[8];
      load8(g + j, gv);
      load8_cg(M + j, mp);
      load8(w + j, wv[c]);
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        m[c][e] = fmaf(a.mu, mp[e], gv[e]);
        dot = fmaf(m[c][e], wv[c][e], dot);
        wsq = fmaf(wv[c][e], wv[c][e], wsq);
      }
      store8(M + j, m[c]);
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) { m[c][e] = 0.f; wv[c][e] = 0.f; }
    }
  }
  dot = block_sum(dot, red);
  if (a.tangent == 2) wsq = block_sum(wsq, red);
  const float coef = tangent_coef(a.tangent, dot, wsq);
  float ss = 0.f;
#pragma unroll
  for (int c = 0; c < 2; ++c)
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      m[c][e] = fmaf(-coef, wv[c][e], m[c][e]);
      ss = fmaf(m[c][e], m[c][e], ss);
    }
  ss = block_sum(ss, red);
  if (a.tangent == 2) {
    float mm = 0.f;
#pragma unroll
    for (int c = 0; c < 2; ++c)
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const float mo = fmaf(coef, wv[c][e], m[c][e]);   // the momentum entry
        mm = fmaf(mo, mo, mm);
      }
    mm = block_sum(mm, red);
    if (ss <= 1e-6f * mm) ss = 0.f;
  }
  const float inv = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
#pragma unroll
  for (int c = 0; c < 2; ++c) {
    const int64_t j = (static_cast<int64_t>(c) * blockDim.x + threadIdx.x) * 8;
    if (j < cols) {
      float v[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) v[e] = m[c][e] * inv;
      store8(psi + j, v);
    }
  }
  if (threadIdx.x == 0) {
    if (ss > 0.f) atomicAdd(&a.count[a.mat_id[b]], 1);
    if (!isfinite(ss) || !isfinite(dot)) raise_flag(a.flags, kFlagNonfinite);
  }
}

// row-active, scalar path (any shape): M is re-read by the thread that wrote it
template <typename TG, typename TW, typename TP>
__global__ void __launch_bounds__(256) k_norm_rows_scalar(const __grid_constant__ NormLaunch a) {
  __shared__ float red[32];
  const int b = blockIdx.y;
  const int64_t row = blockIdx.x;
  const int64_t cols = a.cols;
  const TG* g = static_cast<const TG*>(a.G[b]) + row * cols;
  float* M = a.M[b] + row * cols;
  const TW* w = static_cast<const TW*>(a.W[b]) + row * cols;
  TP* psi = static_cast<TP*>(a.psi[b]) + row * a.psi_ld;
  float dot = 0.f, wsq = 0.f;
  for (int64_t j = threadIdx.x; j < cols; j += blockDim.x) {
    const float m = fmaf(a.mu, M[j], to_f32(g[j]));
    M[j] = m;
    const float wj = to_f32(w[j]);
    dot = fmaf(m, wj, dot);
    wsq = fmaf(wj, wj, wsq);
  }
  dot = block_sum(dot, red);
  if (a.tangent == 2) wsq = block_sum(wsq, red);
  const float coef = tangent_coef(a.tangent, dot, wsq);
  float ss = 0.f;
  float mm = 0.f;
  for (int64_t j = threadIdx.x; j < cols; j += blockDim.x) {
    const float x = fmaf(-coef, to_f32(w[j]), M[j]);
    ss = fmaf(x, x, ss);
    mm = fmaf(M[j], M[j], mm);
  }
  ss = block_sum(ss, red);
  if (a.tangent == 2) {
    mm = block_sum(mm, red);
    if (ss <= 1e-6f * mm) ss = 0.f;
  }
  const float inv = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
  for (int64_t j = threadIdx.x; j < cols; j += blockDim.x)
    psi[j] = from_f32<TP>(fmaf(-coef, to_f32(w[j]), M[j]) * inv);
  if (threadIdx.x == 0) {
    if (ss > 0.f) atomicAdd(&a.count[a.mat_id[b]], 1);
    if (!isfinite(ss) || !isfinite(dot)) raise_flag(a.flags, kFlagNonfinite);
  }
}

// ---------------------------------------------------------------------------
// column-active pass A: momentum + column partial sums
// grid (ceil(cols / 256), nrb, n); thread = (column chunk cc = tid % 32, row lane rl = tid / 32)
// ---------------------------------------------------------------------------
template <typename TG, typename TW, bool VEC>
__global__ void __launch_bounds__(kColThreads) k_norm_cols_stats(const __grid_constant__ NormLaunch a) {
  __shared__ float part[8][3][256];
  const int b = blockIdx.z, rb = blockIdx.y;
  const int cc = threadIdx.x & 31, rl = threadIdx.x >> 5;
  const int64_t rows = a.rows, cols = a.cols;
  const int64_t r0 = static_cast<int64_t>(rb) * kColStatsRB;
  const int64_t r1 = min(r0 + kColStatsRB, rows);
  const TG* g = static_cast<const TG*>(a.G[b]);
  float* M = a.M[b];
  const TW* w = static_cast<const TW*>(a.W[b]);
  float smm[8], smw[8], sww[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) { smm[e] = 0.f; smw[e] = 0.f; sww[e] = 0.f; }
  if (VEC) {
    const int64_t j0 = static_cast<int64_t>(blockIdx.x) * 256 + cc * 8;
    if (j0 < cols) {
#pragma unroll 4
      for (int64_t r = r0 + rl; r < r1; r += 8) {
        float gv[8], mp[8], wv[8];
        load8(g + r * cols + j0, gv);
        load8_cg(M + r * cols + j0, mp);
        load8(w + r * cols + j0, wv);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float m = fmaf(a.mu, mp[e], gv[e]);
          mp[e] = m;
          smm[e] = fmaf(m, m, smm[e]);
          smw[e] = fmaf(m, wv[e], smw[e]);
          sww[e] = fmaf(wv[e], wv[e], sww[e]);
        }
        store8(M + r * cols + j0, mp);
      }
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      part[rl][0][cc * 8 + e] = smm[e];
      part[rl][1][cc * 8 + e] = smw[e];
      part[rl][2][cc * 8 + e] = sww[e];
    }
  } else {
    // scalar: thread handles columns cc + 32 e of the strip
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const int64_t j = static_cast<int64_t>(blockIdx.x) * 256 + cc + 32 * e;
      if (j < cols) {
        for (int64_t r = r0 + rl; r < r1; r += 8) {
          const float m = fmaf(a.mu, M[r * cols + j], to_f32(g[r * cols + j]));
          const float wv = to_f32(w[r * cols + j]);
          M[r * cols + j] = m;
          smm[e] = fmaf(m, m, smm[e]);
          smw[e] = fmaf(m, wv, smw[e]);
          sww[e] = fmaf(wv, wv, sww[e]);
        }
      }
      part[rl][0][cc + 32 * e] = smm[e];
      part[rl][1][cc + 32 * e] = smw[e];
      part[rl][2][cc + 32 * e] = sww[e];
    }
  }
  __syncthreads();
  // fold the 8 row lanes (fp64, fixed order) and write this block's partials
  const int col = threadIdx.x;   // 0..255
  const int64_t j = static_cast<int64_t>(blockIdx.x) * 256 + col;
  if (j < cols) {
    double s0 = 0, s1 = 0, s2 = 0;
#pragma unroll
    for (int l = 0; l < 8; ++l) {
      s0 += part[l][0][col];
      s1 += part[l][1][col];
      s2 += part[l][2][col];
    }
    const int64_t nrb = gridDim.y;
    double* p = a.col_part + ((static_cast<int64_t>(b) * nrb + rb) * cols + j) * 3;
    p[0] = s0; p[1] = s1; p[2] = s2;
  }
}

// column-active fold: per column a_j = <m_j, w_j>, inv_j = 1 / ||x_j||.
// stage 0: both from the pass-A sums (relaxed and no-tangent modes).
// stage 1 (strict): a_j = <m_j, w_j> / ||w_j||^2 only.
// stage 2 (strict): ||x_j||^2 from the direct sums of k_norm_cols_xsq (slot 1),
// ||m_j||^2 from pass A (slot 0), a_j kept.
__global__ void __launch_bounds__(256) k_norm_cols_final(const __grid_constant__ NormLaunch a, int nrb, int stage) {
  __shared__ float red[32];
  const int b = blockIdx.y;
  const int64_t cols = a.cols;
  const int64_t j = static_cast<int64_t>(blockIdx.x) * 256 + threadIdx.x;
  float nz = 0.f;
  if (j < cols) {
    double s0 = 0, s1 = 0, s2 = 0;
    const double* p = a.col_part + (static_cast<int64_t>(b) * nrb * cols + j) * 3;
    for (int rb = 0; rb < nrb; ++rb) {
      s0 += p[0]; s1 += p[1]; s2 += p[2];
      p += cols * 3;
    }
    float2* out = a.col_coef + static_cast<int64_t>(b) * cols + j;
    if (stage == 1) {
      // strict: only the projection coefficient; the norm comes from the direct pass
      *out = make_float2(s2 > 0.0 ? static_cast<float>(s1 / s2) : 0.f, 0.f);
    } else {
      // relaxed: a = S_mw, ||x||^2 = S_mm - a^2 (2 - S_ww); none: a = 0,
      // ||x||^2 = S_mm; strict (stage 2): S_xx summed directly
      double aa, d2;
      if (stage == 2) {
        aa = out->x;
        d2 = s1;
        if (d2 <= 1e-6 * s0) d2 = 0.0;   // parallel to the weight column: no tangent part
      }
      else if (a.tangent == 0) { aa = s1; d2 = s0 - aa * aa * (2.0 - s2); }
      else { aa = 0.0; d2 = s0; }
      if (!(d2 > 0.0)) d2 = (d2 == d2) ? 0.0 : d2;    // clamp rounding below zero, keep NaN
      const float inv = d2 > 0.0 ? static_cast<float>(1.0 / sqrt(d2)) : 0.f;
      *out = make_float2(static_cast<float>(aa), inv);
      nz = d2 > 0.0 ? 1.f : 0.f;
      if (!isfinite(d2) || !isfinite(aa)) raise_flag(a.flags, kFlagNonfinite);
    }
  }
  nz = block_sum(nz, red);
  if (threadIdx.x == 0 && nz > 0.f) atomicAdd(&a.count[a.mat_id[b]], static_cast<int>(nz));
}

// strict tangent, column-active: ||x_j||^2 of this block's rows summed from
// x_ij = m_ij - a_j w_ij itself (no cancellation), into slot 1 of the
// block's partials (the <m, w> sums, already folded into a_j).
// grid and thread layout as pass A.
template <typename TW, bool VEC>
__global__ void __launch_bounds__(kColThreads) k_norm_cols_xsq(const __grid_constant__ NormLaunch a) {
  __shared__ float part[8][256];
  const int b = blockIdx.z, rb = blockIdx.y;
  const int cc = threadIdx.x & 31, rl = threadIdx.x >> 5;
  const int64_t rows = a.rows, cols = a.cols;
  const int64_t r0 = static_cast<int64_t>(rb) * kColStatsRB;
  const int64_t r1 = min(r0 + kColStatsRB, rows);
  const float* M = a.M[b];
  const TW* w = static_cast<const TW*>(a.W[b]);
  const float2* coef = a.col_coef + static_cast<int64_t>(b) * cols;
  if (VEC) {
    const int64_t j0 = static_cast<int64_t>(blockIdx.x) * 256 + cc * 8;
    float sx[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) sx[e] = 0.f;
    if (j0 < cols) {
      float ca[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) ca[e] = coef[j0 + e].x;
      for (int64_t r = r0 + rl; r < r1; r += 8) {
        float mv[8], wv[8];
        load8(M + r * cols + j0, mv);
        load8(w + r * cols + j0, wv);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float x = fmaf(-ca[e], wv[e], mv[e]);
          sx[e] = fmaf(x, x, sx[e]);
        }
      }
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) part[rl][cc * 8 + e] = sx[e];
  } else {
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const int64_t j = static_cast<int64_t>(blockIdx.x) * 256 + cc + 32 * e;
      float sx = 0.f;
      if (j < cols) {
        const float cj = coef[j].x;
        for (int64_t r = r0 + rl; r < r1; r += 8) {
          const float x = fmaf(-cj, to_f32(w[r * cols + j]), M[r * cols + j]);
          sx = fmaf(x, x, sx);
        }
      }
      part[rl][cc + 32 * e] = sx;
    }
  }
  __syncthreads();
  const int col = threadIdx.x;
  const int64_t j = static_cast<int64_t>(blockIdx.x) * 256 + col;
  if (j < cols) {
    double s = 0;
#pragma unroll
    for (int l = 0; l < 8; ++l) s += part[l][col];
    a.col_part[((static_cast<int64_t>(b) * gridDim.y + rb) * cols + j) * 3 + 1] = s;
  }
}

// column-active pass B: Psi_ij = (m_ij - a_j w_ij) * inv_j
template <typename TW, typename TP, bool VEC>
__global__ void __launch_bounds__(kColThreads) k_norm_cols_apply(const __grid_constant__ NormLaunch a) {
  const int b = blockIdx.z, rb = blockIdx.y;
  const int cc = threadIdx.x & 31, rl = threadIdx.x >> 5;
  const int64_t rows = a.rows, cols = a.cols;
  const int64_t r0 = static_cast<int64_t>(rb) * kColApplyRB;
  const int64_t r1 = min(r0 + kColApplyRB, rows);
  const float* M = a.M[b];
  const TW* w = static_cast<const TW*>(a.W[b]);
  TP* psi = static_cast<TP*>(a.psi[b]);
  const float2* coef = a.col_coef + static_cast<int64_t>(b) * cols;
  if (VEC) {
    const int64_t j0 = static_cast<int64_t>(blockIdx.x) * 256 + cc * 8;
    if (j0 >= cols) return;
    float ca[8], ci[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) { const float2 c = coef[j0 + e]; ca[e] = c.x; ci[e] = c.y; }
    for (int64_t r = r0 + rl; r < r1; r += 8) {
      float mv[8], wv[8];
      load8(M + r * cols + j0, mv);
      load8(w + r * cols + j0, wv);
#pragma unroll
      for (int e = 0; e < 8; ++e) mv[e] = fmaf(-ca[e], wv[e], mv[e]) * ci[e];
      store8(psi + r * a.psi_ld + j0, mv);
    }
  } else {
    for (int e = 0; e < 8; ++e) {
      const int64_t j = static_cast<int64_t>(blockIdx.x) * 256 + cc + 32 * e;
      if (j >= cols) break;
      const float2 c = coef[j];
      for (int64_t r = r0 + rl; r < r1; r += 8)
        psi[r * a.psi_ld + j] = from_f32<TP>(fmaf(-c.x, to_f32(w[r * cols + j]), M[r * cols + j]) * c.y);
    }
  }
}

// ---------------------------------------------------------------------------
// "Row+Column/Step" (orientation 3, Table 5b): after the row normalization,
// the columns of Psi (stored layout, row stride psi_ld) are normalized in
// place.  Pass 1 sums psi^2 per (block of kColStatsRB rows, column) into fp64
// partials; a fold (one CTA per matrix, fixed order) writes 1 / ||column||
// and sets count[] to the number of nonzero columns (then ||Psi||_F^2);
// pass 2 scales.
// ---------------------------------------------------------------------------
template <typename TP>
__global__ void __launch_bounds__(256) k_psi_colsq(const __grid_constant__ NormLaunch a) {
  const int b = blockIdx.z, rb = blockIdx.y;
  const int64_t j = static_cast<int64_t>(blockIdx.x) * 256 + threadIdx.x;
  if (j >= a.cols) return;
  const TP* psi = static_cast<const TP*>(a.psi[b]);
  const int64_t r0 = static_cast<int64_t>(rb) * kColStatsRB, r1 = min(r0 + kColStatsRB, a.rows);
  float s = 0.f;
  for (int64_t r = r0; r < r1; ++r) {
    const float v = to_f32(psi[r * a.psi_ld + j]);
    s = fmaf(v, v, s);
  }
  a.col_part[(static_cast<int64_t>(b) * gridDim.y + rb) * a.cols + j] = s;
}

__global__ void __launch_bounds__(256) k_psi_colfold(const __grid_constant__ NormLaunch a, int nrb) {
  __shared__ float red[32];
  const int b = blockIdx.x;
  float nz = 0.f;
  for (int64_t j = threadIdx.x; j < a.cols; j += blockDim.x) {
    double s = 0;
    for (int rb = 0; rb < nrb; ++rb) s += a.col_part[(static_cast<int64_t>(b) * nrb + rb) * a.cols + j];
    const float inv = s > 0.0 ? static_cast<float>(1.0 / sqrt(s)) : 0.f;
    a.col_coef[static_cast<int64_t>(b) * a.cols + j] = make_float2(0.f, inv);
    nz += s > 0.0 ? 1.f : 0.f;
  }
  nz = block_sum(nz, red);
  if (threadIdx.x == 0) a.count[a.mat_id[b]] = static_cast<int>(nz);
}

template <typename TP>
__global__ void __launch_bounds__(256) k_psi_colscale(const __grid_constant__ NormLaunch a) {
  const int b = blockIdx.z;
  const int64_t j = static_cast<int64_t>(blockIdx.x) * 256 + threadIdx.x;
  if (j >= a.cols) return;
  const float inv = a.col_coef[static_cast<int64_t>(b) * a.cols + j].y;
  TP* psi = static_cast<TP*>(a.psi[b]);
  const int64_t r0 = static_cast<int64_t>(blockIdx.y) * kColApplyRB, r1 = min(r0 + kColApplyRB, a.rows);
  for (int64_t r = r0; r < r1; ++r) psi[r * a.psi_ld + j] = from_f32<TP>(to_f32(psi[r * a.psi_ld + j]) * inv);
}

cudaError_t launch_normalize_psi_cols(const NormLaunch& a, cudaStream_t s) {
  if (a.n <= 0 || a.rows <= 0 || a.cols <= 0) return cudaSuccess;
  const int nrb = static_cast<int>(cdiv(a.rows, kColStatsRB));
  const unsigned cb = static_cast<unsigned>(cdiv(a.cols, 256));
  if (a.psi_dtype == 1) k_psi_colsq<bf16><<<dim3(cb, nrb, a.n), 256, 0, s>>>(a);
  else k_psi_colsq<float><<<dim3(cb, nrb, a.n), 256, 0, s>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_psi_colfold<<<a.n, 256, 0, s>>>(a, nrb);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const dim3 g2(cb, static_cast<unsigned>(cdiv(a.rows, kColApplyRB)), a.n);
  if (a.psi_dtype == 1) k_psi_colscale<bf16><<<g2, 256, 0, s>>>(a);
  else k_psi_colscale<float><<<g2, 256, 0, s>>>(a);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------
template <typename F>
static cudaError_t dispatch3(int g, int w, int p, F&& f) {
  // g, w, p: 0 = f32, 1 = bf16
  if (g == 0 && w == 0 && p == 0) return f((float*)0, (float*)0, (float*)0);
  if (g == 0 && w == 0 && p == 1) return f((float*)0, (float*)0, (bf16*)0);
  if (g == 0 && w == 1 && p == 0) return f((float*)0, (bf16*)0, (float*)0);
  if (g == 0 && w == 1 && p == 1) return f((float*)0, (bf16*)0, (bf16*)0);
  if (g == 1 && w == 0 && p == 0) return f((bf16*)0, (float*)0, (float*)0);
  if (g == 1 && w == 0 && p == 1) return f((bf16*)0, (float*)0, (bf16*)0);
  if (g == 1 && w == 1 && p == 0) return f((bf16*)0, (bf16*)0, (float*)0);
  return f((bf16*)0, (bf16*)0, (bf16*)0);
}

cudaError_t launch_normalize_rows(const NormLaunch& a, cudaStream_t s) {
  if (a.n <= 0 || a.rows <= 0 || a.cols <= 0) return cudaSuccess;
  const bool vec = (a.cols % 8 == 0) && (a.psi_ld % 8 == 0) && a.cols <= 16 * 1024;
  const dim3 grid(static_cast<unsigned>(a.rows), static_cast<unsigned>(a.n));
  return dispatch3(a.g_dtype, a.w_dtype, a.psi_dtype, [&](auto* tg, auto* tw, auto* tp) {
    using TG = std::remove_pointer_t<decltype(tg)>;
    using TW = std::remove_pointer_t<decltype(tw)>;
    using TP = std::remove_pointer_t<decltype(tp)>;
    if (vec) {
      int threads = static_cast<int>(round_up(cdiv(a.cols, 16), 32));
      threads = threads < 32 ? 32 : threads;
      k_norm_rows_vec<TG, TW, TP><<<grid, threads, 0, s>>>(a);
    } else {
      k_norm_rows_scalar<TG, TW, TP><<<grid, 256, 0, s>>>(a);
    }
    return cudaGetLastError();
  });
}

cudaError_t launch_normalize_cols(const NormLaunch& a, cudaStream_t s) {
  if (a.n <= 0 || a.rows <= 0 || a.cols <= 0) return cudaSuccess;
  const bool vec = (a.cols % 8 == 0) && (a.psi_ld % 8 == 0);
  const int nrb = static_cast<int>(cdiv(a.rows, kColStatsRB));
  const dim3 grid(static_cast<unsigned>(cdiv(a.cols, 256)), static_cast<unsigned>(nrb),
                  static_cast<unsigned>(a.n));
  const dim3 grid_b(grid.x, static_cast<unsigned>(cdiv(a.rows, kColApplyRB)), static_cast<unsigned>(a.n));
  return dispatch3(a.g_dtype, a.w_dtype, a.psi_dtype, [&](auto* tg, auto* tw, auto* tp) {
    using TG = std::remove_pointer_t<decltype(tg)>;
    using TW = std::remove_pointer_t<decltype(tw)>;
    using TP = std::remove_pointer_t<decltype(tp)>;
    if (vec) k_norm_cols_stats<TG, TW, true><<<grid, kColThreads, 0, s>>>(a);
    else k_norm_cols_stats<TG, TW, false><<<grid, kColThreads, 0, s>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (a.tangent == 2) {
      // strict: the coefficient first, then ||x_j||^2 summed from x itself
      k_norm_cols_final<<<dim3(grid.x, a.n), 256, 0, s>>>(a, nrb, 1);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
      if (vec) k_norm_cols_xsq<TW, true><<<grid, kColThreads, 0, s>>>(a);
      else k_norm_cols_xsq<TW, false><<<grid, kColThreads, 0, s>>>(a);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
      k_norm_cols_final<<<dim3(grid.x, a.n), 256, 0, s>>>(a, nrb, 2);
    } else {
      k_norm_cols_final<<<dim3(grid.x, a.n), 256, 0, s>>>(a, nrb, 0);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (vec) k_norm_cols_apply<TW, TP, true><<<grid_b, kColThreads, 0, s>>>(a);
    else k_norm_cols_apply<TW, TP, false><<<grid_b, kColThreads, 0, s>>>(a);
    return cudaGetLastError();
  });
}

}  // namespace normpre
