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
// The eigendecomposition never forms Gamma.  Its nonzero eigenvalues are the
// squared singular values of Psi, and its eigenvectors Psi's singular
// vectors on the active side, so the solver is a one-sided block Jacobi SVD
// (Hestenes' method on column blocks) of the stored Psi:
//   * Z (L x s) holds the shorter side of Psi as columns (s = min(rows, cols),
//     L = max), zero-padded to s_pad, a multiple of 64 columns;
//   * a sweep pairs the 32-column blocks of Z round-robin (s_pad / 32 - 1
//     rounds of disjoint pairs, one CTA per pair): the CTA forms the 64 x 64
//     Gram matrix of its two blocks (fp32 per 64-row chunk, fp64 across
//     chunks), diagonalizes it by a parallel cyclic Jacobi in shared memory,
//     and rotates its 64 columns of Z by the eigenvectors;
//   * a pair whose columns are already orthogonal to 1e-5 (relative to their
//     norms, or 1e-6 of the mean eigenvalue in absolute terms, the accuracy
//     fp32 rotations leave small columns) is left alone; a sweep without any
//     rotation ends the iteration (CTAs of later sweeps return at once), at
//     most kOjMaxSweeps sweeps;
//   * then Z V = U Sigma: lambda_i = ||z_i||^2, and the eigenvector of
//     lambda_i is z_i / sigma_i when Gamma lives on Z's long side (m_a = L),
//     else Psi_a z_i / lambda_i (one contraction with Psi for the selected
//     columns); Gamma's other m_a - s eigenvalues are zero.
// Every matrix of a group is processed by the same launches.
#include <algorithm>
#include <string>

#include "common.cuh"
#include "internal.h"

namespace normpre {

namespace {

constexpr int kOjB = 32;               // columns per block
constexpr int kOjP = 2 * kOjB;         // columns of a block pair
constexpr int kOjRows = 64;            // rows per chunk of the Gram and rotation passes
constexpr int kOjMaxSweeps = kExactFlagRows - 1;
constexpr float kOjTol = 1e-5f;        // |<z_i, z_j>| <= tol ||z_i|| ||z_j||: orthogonal enough
constexpr float kOjAbsTol = 1e-6f;     // ... or |<z_i, z_j>| <= abs_tol * (mean eigenvalue)
constexpr int kOjLdA = kOjP + 1;       // row stride of the 64 x 64 Jacobi matrices
constexpr int kOjLdX = kOjP + 4;       // row stride of a chunk (16-byte rows)
constexpr int kOjSelectMax = 16384;    // eigenvalues one selection CTA sorts (power of two)
constexpr size_t kOjSmem = sizeof(float) * (3 * kOjP * kOjLdA + kOjRows * kOjLdX + kOjP * kOjLdX) + 64 * 16;

// Z: column c (c < s) of matrix b = row c of Psi (when rows <= cols) or column
// c of Psi, at z + (b * s_pad + c) * lp; columns s..s_pad-1 and rows L..lp-1
// are zero.  32 x 32 tiles through shared memory, both sides coalesced.
struct OjLoadArgs {
  const float* psi; int64_t psi_bs, ld;
  float* z;
  int64_t s, s_pad, L, lp;
  int cols_are_rows;
};
__global__ void __launch_bounds__(256) k_oj_load(const __grid_constant__ OjLoadArgs a) {
  __shared__ float t[32][33];
  const int b = blockIdx.z;
  const int64_t c0 = static_cast<int64_t>(blockIdx.y) * 32, r0 = static_cast<int64_t>(blockIdx.x) * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;   // 32 x 8
  const float* psi = a.psi + b * a.psi_bs;
  for (int k = ty; k < 32; k += 8) {
    // element (column c of Z, row r of Z)
    if (a.cols_are_rows) {
      const int64_t c = c0 + k, r = r0 + tx;              // Psi[c][r]: r contiguous
      t[k][tx] = (c < a.s && r < a.L) ? psi[c * a.ld + r] : 0.f;
    } else {
      const int64_t r = r0 + k, c = c0 + tx;              // Psi[r][c]: c contiguous
      t[tx][k] = (c < a.s && r < a.L) ? psi[r * a.ld + c] : 0.f;
    }
  }
  __syncthreads();
  float* z = a.z + static_cast<int64_t>(b) * a.s_pad * a.lp;
  for (int k = ty; k < 32; k += 8) {
    const int64_t c = c0 + k, r = r0 + tx;
    if (c < a.s_pad && r < a.lp) z[c * a.lp + r] = t[k][tx];
  }
}

// Rotation of the symmetric pair (p, q): J = [[c, s], [-s, c]] on columns
// (p, q) makes J^T [[app, apq], [apq, aqq]] J diagonal (Golub and Van Loan,
// symmetric Schur decomposition of a 2 x 2 block).
__device__ __forceinline__ void oj_rot(float app, float aqq, float apq, float& c, float& s) {
  if (!(fabsf(apq) > 0.f)) { c = 1.f; s = 0.f; return; }
  const float tau = (aqq - app) / (2.f * apq);
  const float t = (tau >= 0.f ? 1.f : -1.f) / (fabsf(tau) + sqrtf(fmaf(tau, tau, 1.f)));
  c = 1.f / sqrtf(fmaf(t, t, 1.f));
  s = t * c;
}

// Loads rows [r0, r0 + 64) of the pair's 64 columns into X[row][col].
__device__ __forceinline__ void oj_load_chunk(const float* zb, int I, int J, int64_t lp, int64_t r0, float* X) {
  for (int e = threadIdx.x; e < kOjP * (kOjRows / 4); e += blockDim.x) {
    const int col = e / (kOjRows / 4), r4 = 4 * (e % (kOjRows / 4));
    const int zc = col < kOjB ? I * kOjB + col : J * kOjB + col - kOjB;
    const float4 v = *reinterpret_cast<const float4*>(zb + zc * lp + r0 + r4);
    X[(r4 + 0) * kOjLdX + col] = v.x;
    X[(r4 + 1) * kOjLdX + col] = v.y;
    X[(r4 + 2) * kOjLdX + col] = v.z;
    X[(r4 + 3) * kOjLdX + col] = v.w;
  }
}

struct OjRoundArgs {
  float* z;
  int64_t s_pad, lp;
  int nb;                // blocks of 32 columns (even)
  int round, sweep;
  int* flag;             // [kOjMaxSweeps][batch]: 1 when the sweep rotated a pair
  int batch;
  const int* count;      // m' per matrix id: ||Psi||_F^2 (its active rows are unit vectors)
  const int* mat_ids;
  int64_t s;             // Z's true column count (mean eigenvalue = m' / s)
};
// One CTA per (block pair, matrix) of one round of one sweep; 256 threads.
__global__ void __launch_bounds__(256) k_oj_round(const __grid_constant__ OjRoundArgs a) {
  extern __shared__ float4 oj_smem4[];
  float* A = reinterpret_cast<float*>(oj_smem4);      // [64][65] Gram, then Jacobi copy 1
  float* A2 = A + kOjP * kOjLdA;                      // Jacobi copy 2
  float* V = A2 + kOjP * kOjLdA;                      // [64][65] eigenvectors
  float* X = V + kOjP * kOjLdA;                       // [64 rows][68] chunk
  float* Vx = X + kOjRows * kOjLdX;                   // [64][68] eigenvectors, 16-byte rows
  float4* rot = reinterpret_cast<float4*>(Vx + kOjP * kOjLdX);   // [32]
  __shared__ double dred[8];
  __shared__ float fred[8];
  __shared__ int skip_s;
  const int b = blockIdx.y, pr = blockIdx.x, tid = threadIdx.x;
  if (a.sweep > 0 && a.flag[(a.sweep - 1) * a.batch + b] == 0) return;   // converged
  // round-robin pairing of the nb blocks: block 0 stays, the others rotate
  const int n1 = a.nb - 1;
  int I, J;
  if (pr == 0) { I = 0; J = 1 + (a.round % n1); }
  else { I = 1 + (pr + a.round) % n1; J = 1 + (n1 - pr + a.round) % n1; }
  float* zb = a.z + static_cast<int64_t>(b) * a.s_pad * a.lp;
  const int tr = tid >> 4, tc = tid & 15;            // 4 x 4 output tile (rows 4 tr, cols 4 tc)

  // ---- Gram of the 64 columns: fp32 per chunk, fp64 across chunks ----
  double g64[4][4] = {};
  for (int64_t r0 = 0; r0 < a.lp; r0 += kOjRows) {
    const int nr = static_cast<int>(a.lp - r0 < kOjRows ? a.lp - r0 : kOjRows);
    __syncthreads();
    oj_load_chunk(zb, I, J, a.lp, r0, X);
    __syncthreads();
    float acc[4][4] = {};
    for (int i = 0; i < nr; ++i) {
      const float4 p = *reinterpret_cast<const float4*>(X + i * kOjLdX + 4 * tr);
      const float4 q = *reinterpret_cast<const float4*>(X + i * kOjLdX + 4 * tc);
      const float pa[4] = {p.x, p.y, p.z, p.w}, qa[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(pa[u], qa[v], acc[u][v]);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int v = 0; v < 4; ++v) g64[u][v] += acc[u][v];
  }
#pragma unroll
  for (int u = 0; u < 4; ++u)
#pragma unroll
    for (int v = 0; v < 4; ++v) A[(4 * tr + u) * kOjLdA + 4 * tc + v] = static_cast<float>(g64[u][v]);
  __syncthreads();

  // ---- already orthogonal to kOjTol? (columns of zero norm do not count) ----
  float dmax = 0.f;
  for (int i = tid; i < kOjP; i += blockDim.x) dmax = fmaxf(dmax, A[i * kOjLdA + i]);
  dmax = warp_max(dmax);
  if ((tid & 31) == 0) fred[tid >> 5] = dmax;
  __syncthreads();
  dmax = 0.f;
  for (int w = 0; w < 8; ++w) dmax = fmaxf(dmax, fred[w]);
  // columns below 1e-12 ||Psi||_F^2 are numerically zero (what a rank-deficient
  // Psi leaves after rotation): no orthogonality is asked of them
  const float fro2 = fmaxf(static_cast<float>(a.count[a.mat_ids[b]]), 1.f);
  const float zero_norm = fmaxf(1e-30f * dmax, 1e-12f * fro2);
  // fp32 rotations leave a column about u sqrt(lambda_max / lambda_i) of
  // relative error, so small columns cannot become orthogonal relative to
  // their own norms; only the eigenvectors of large eigenvalues are used, and
  // the small eigenvalues need absolute accuracy: a pair also counts as done
  // below kOjAbsTol of the mean eigenvalue
  const float abs_tol = kOjAbsTol * fro2 / static_cast<float>(a.s);
  float worst = 0.f;
  for (int e = tid; e < kOjP * kOjP; e += blockDim.x) {
    const int i = e / kOjP, j = e % kOjP;
    if (i == j) continue;
    const float aii = A[i * kOjLdA + i], ajj = A[j * kOjLdA + j];
    const float aij = fabsf(A[i * kOjLdA + j]);
    if (aii > zero_norm && ajj > zero_norm && aij > abs_tol) worst = fmaxf(worst, aij * rsqrtf(aii * ajj));
  }
  worst = warp_max(worst);
  __syncthreads();
  if ((tid & 31) == 0) fred[tid >> 5] = worst;
  __syncthreads();
  if (tid == 0) {
    float w = 0.f;
    for (int k = 0; k < 8; ++k) w = fmaxf(w, fred[k]);
    skip_s = !(w > kOjTol) || !(dmax > zero_norm);
    if (!skip_s) a.flag[a.sweep * a.batch + b] = 1;
  }
  __syncthreads();
  if (skip_s) return;

  // ---- parallel cyclic Jacobi of the 64 x 64 Gram matrix ----
  for (int e = tid; e < kOjP * kOjLdA; e += blockDim.x) V[e] = ((e % kOjLdA) == (e / kOjLdA)) ? 1.f : 0.f;
  double frob = 0.0;
  for (int e = tid; e < kOjP * kOjP; e += blockDim.x) {
    const float x = A[(e / kOjP) * kOjLdA + e % kOjP];
    frob += static_cast<double>(x) * x;
  }
  frob = warp_sum(frob);
  if ((tid & 31) == 0) dred[tid >> 5] = frob;
  __syncthreads();
  frob = 0.0;
  for (int w = 0; w < 8; ++w) frob += dred[w];
  float* cur = A;
  float* nxt = A2;
  int pk = (tid == 0) ? 0 : tid, qk = kOjP - 1 - tid;   // players of pair tid (tid < 32)
  double off = frob, prev = frob;
  for (int sw = 0; sw < 10; ++sw) {
    for (int step = 0; step < kOjP - 1; ++step) {
      if (tid < kOjB) {
        const int i = min(pk, qk), j = max(pk, qk);
        float c, s;
        oj_rot(cur[i * kOjLdA + i], cur[j * kOjLdA + j], cur[i * kOjLdA + j], c, s);
        rot[tid] = make_float4(c, s, __int_as_float(i), __int_as_float(j));
        if (tid != 0) pk = (pk == kOjP - 1) ? 1 : pk + 1;
        qk = (qk == kOjP - 1) ? 1 : qk + 1;
      }
      __syncthreads();
      // J^T A J by 2 x 2 blocks (rows of pair k1, columns of pair k2) into the other copy
      for (int e = tid; e < kOjB * kOjB; e += blockDim.x) {
        const int k1 = e / kOjB, k2 = e % kOjB;
        const float4 r1 = rot[k1], r2 = rot[k2];
        const int i = __float_as_int(r1.z), j = __float_as_int(r1.w);
        const int i2 = __float_as_int(r2.z), j2 = __float_as_int(r2.w);
        const float a00 = cur[i * kOjLdA + i2], a01 = cur[i * kOjLdA + j2];
        const float a10 = cur[j * kOjLdA + i2], a11 = cur[j * kOjLdA + j2];
        const float u0 = r2.x * a00 - r2.y * a01, w0 = r2.y * a00 + r2.x * a01;
        const float u1 = r2.x * a10 - r2.y * a11, w1 = r2.y * a10 + r2.x * a11;
        nxt[i * kOjLdA + i2] = r1.x * u0 - r1.y * u1;
        nxt[j * kOjLdA + i2] = r1.y * u0 + r1.x * u1;
        nxt[i * kOjLdA + j2] = r1.x * w0 - r1.y * w1;
        nxt[j * kOjLdA + j2] = r1.y * w0 + r1.x * w1;
      }
      // V <- V J: (row, pair) items
      for (int e = tid; e < kOjP * kOjB; e += blockDim.x) {
        const int row = e / kOjB, k = e % kOjB;
        const float4 r = rot[k];
        const int i = __float_as_int(r.z), j = __float_as_int(r.w);
        const float vi = V[row * kOjLdA + i], vj = V[row * kOjLdA + j];
        V[row * kOjLdA + i] = r.x * vi - r.y * vj;
        V[row * kOjLdA + j] = r.y * vi + r.x * vj;
      }
      __syncthreads();
      float* t = cur; cur = nxt; nxt = t;
    }
    double so = 0.0;
    for (int e = tid; e < kOjP * kOjP; e += blockDim.x) {
      const int i = e / kOjP, j = e % kOjP;
      if (i != j) so += static_cast<double>(cur[i * kOjLdA + j]) * cur[i * kOjLdA + j];
    }
    so = warp_sum(so);
    __syncthreads();
    if ((tid & 31) == 0) dred[tid >> 5] = so;
    __syncthreads();
    prev = off;
    off = 0.0;
    for (int w = 0; w < 8; ++w) off += dred[w];
    // the fp32 floor: Jacobi converges quadratically, so a sweep that no
    // longer halves a tiny off-diagonal mass has reached rounding
    if (off <= 1e-14 * frob || (off <= 1e-10 * frob && off > 0.5 * prev)) break;
  }
  // V is orthogonal only to ~1e-6 after the fp32 rotations, and every round
  // applies it to the columns, whose norms (the singular values) would drift
  // by as much; one polar correction V <- V - V E / 2 with E = V^T V - I
  // (E summed with error-free products and compensated additions) leaves V
  // orthogonal to fp32 rounding.  E goes to the free Jacobi copy, the
  // corrected V to the 16-byte-row copy the rotation pass reads.
  __syncthreads();
  float* E = (cur == A) ? A2 : A;
  for (int e = tid; e < kOjP * kOjP; e += blockDim.x) {
    const int i = e / kOjP, j = e % kOjP;
    float hi = (i == j) ? -1.f : 0.f, lo = 0.f;
    for (int k = 0; k < kOjP; ++k) {
      const float x = V[k * kOjLdA + i], y = V[k * kOjLdA + j];
      const float pr = x * y;
      const float pe = fmaf(x, y, -pr);          // x y = pr + pe exactly
      const float sm = hi + pr;                  // two-sum of hi and pr
      const float bv = sm - hi;
      lo += ((hi - (sm - bv)) + (pr - bv)) + pe;
      hi = sm;
    }
    E[i * kOjLdA + j] = hi + lo;
  }
  __syncthreads();
  {
    float acc[4][4] = {};
    for (int k = 0; k < kOjP; ++k) {
      float ev[4];
#pragma unroll
      for (int w = 0; w < 4; ++w) ev[w] = E[k * kOjLdA + 4 * tc + w];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float v = V[(4 * tr + u) * kOjLdA + k];
#pragma unroll
        for (int w = 0; w < 4; ++w) acc[u][w] = fmaf(v, ev[w], acc[u][w]);
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int w = 0; w < 4; ++w)
        Vx[(4 * tr + u) * kOjLdX + 4 * tc + w] = fmaf(-0.5f, acc[u][w], V[(4 * tr + u) * kOjLdA + 4 * tc + w]);
  }

  // ---- rotate the pair's columns: Z[:, pair] <- Z[:, pair] V ----
  for (int64_t r0 = 0; r0 < a.lp; r0 += kOjRows) {
    const int nr = static_cast<int>(a.lp - r0 < kOjRows ? a.lp - r0 : kOjRows);
    __syncthreads();
    oj_load_chunk(zb, I, J, a.lp, r0, X);
    __syncthreads();
    float out[4][4] = {};
    for (int k = 0; k < kOjP; ++k) {
      const float4 v = *reinterpret_cast<const float4*>(Vx + k * kOjLdX + 4 * tc);
      const float va[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float x = X[(4 * tr + u) * kOjLdX + k];
#pragma unroll
        for (int w = 0; w < 4; ++w) out[u][w] = fmaf(x, va[w], out[u][w]);
      }
    }
    // thread (tr, tc): rows 4 tr .. 4 tr + 3 of columns 4 tc .. 4 tc + 3
    if (4 * tr < nr) {
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        const int col = 4 * tc + w;
        const int zc = col < kOjB ? I * kOjB + col : J * kOjB + col - kOjB;
        *reinterpret_cast<float4*>(zb + zc * a.lp + r0 + 4 * tr) =
            make_float4(out[0][w], out[1][w], out[2][w], out[3][w]);
      }
    }
  }
}

// lambda_c = ||z_c||^2 (fp64 sums), one warp per column
struct OjNormArgs {
  const float* z;
  int64_t s, s_pad, lp;
  float* lam;            // [batch][s_pad]
};
__global__ void __launch_bounds__(256) k_oj_norms(const __grid_constant__ OjNormArgs a) {
  const int b = blockIdx.y;
  const int64_t c = static_cast<int64_t>(blockIdx.x) * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (c >= a.s_pad) return;
  const float* col = a.z + (static_cast<int64_t>(b) * a.s_pad + c) * a.lp;
  double acc = 0.0;
  for (int64_t r = lane; r < a.lp; r += 32) acc += static_cast<double>(col[r]) * col[r];
  acc = warp_sum(acc);
  if (lane == 0) a.lam[static_cast<int64_t>(b) * a.s_pad + c] = c < a.s ? static_cast<float>(acc) : -1.f;
}

// One CTA per matrix: the s eigenvalues sorted (bitonic, descending, ties by
// lower column), Gamma's spectrum (the s values, then m_a - s zeros), the
// selection C, K, the Ritz slots, the statistics, the energies and the
// column of Z behind each selected eigenvalue.
struct OjSelectArgs {
  const float* lam; int64_t s, s_pad, m_a, n_a;
  int npow;              // power of two >= s_pad
  int l, rank, k_orient;
  const int* flag; int sweeps_flag_row, batch;   // flag row of the last sweep
  float* eig_all; int64_t eig_bs;
  float* ritz; int64_t ritz_bs;
  float* z; float* kmat; int64_t sq;
  float* stats;
  int* sel; int64_t sel_bs;                      // [l] column of Z per selected slot (-1: none)
  float* sel_lam;                                // [l] its eigenvalue
  double* diag; const int* mat_ids;
  const int* count;
  int* flags;
};
__global__ void __launch_bounds__(1024) k_oj_select(const __grid_constant__ OjSelectArgs a) {
  extern __shared__ float4 sel_smem4[];
  float* key = reinterpret_cast<float*>(sel_smem4);
  int* idx = reinterpret_cast<int*>(key + a.npow);
  __shared__ double red[32];
  __shared__ int nc_s;
  const int b = blockIdx.x, tid = threadIdx.x, nt = blockDim.x;
  const float* lam = a.lam + static_cast<int64_t>(b) * a.s_pad;
  for (int i = tid; i < a.npow; i += nt) {
    key[i] = i < a.s ? lam[i] : -1.f;    // padding sorts last (eigenvalues are >= 0)
    idx[i] = i;
  }
  __syncthreads();
  // bitonic sort, descending by key, ascending index among equal keys
  for (int k = 2; k <= a.npow; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = tid; i < a.npow; i += nt) {
        const int p = i ^ j;
        if (p > i) {
          const bool desc = (i & k) == 0;
          const float ki = key[i], kp = key[p];
          const int ii = idx[i], ip = idx[p];
          // "i before p" in the final order
          const bool ordered = (ki > kp) || (ki == kp && ii < ip);
          if (desc ? !ordered : ordered) {
            key[i] = kp; key[p] = ki;
            idx[i] = ip; idx[p] = ii;
          }
        }
      }
      __syncthreads();
    }
  }
  float* eig = a.eig_all + b * a.eig_bs;
  for (int64_t i = tid; i < a.m_a; i += nt) eig[i] = i < a.s ? fmaxf(key[i], 0.f) : 0.f;
  const int l = a.l, rr = min(a.rank, l);
  if (tid == 0) {
    int nc = 0;
    for (int c = 0; c < rr && c < a.s; ++c) {
      if (!(key[c] > 1.f)) break;
      ++nc;
    }
    nc_s = nc;
  }
  __syncthreads();
  const int nc = nc_s;
  float* zz = a.z + b * a.sq;
  float* km = a.kmat + b * a.sq;
  for (int e = tid; e < l * l; e += nt) {
    const int r = e / l, c = e % l;
    zz[e] = (r == c) ? 1.f : 0.f;
    km[e] = (r == c && c < nc) ? rsqrtf(key[c]) - 1.f : 0.f;
  }
  for (int c = tid; c < l; c += nt) {
    a.ritz[b * a.ritz_bs + c] = c < a.s ? fmaxf(key[c], 0.f) : 0.f;
    a.sel[b * a.sel_bs + c] = c < nc ? idx[c] : -1;
    a.sel_lam[b * a.sel_bs + c] = c < nc ? key[c] : 0.f;
  }
  // sums over the spectrum in fp64: the excess of C and the three energies
  // (the m_a - s zero eigenvalues add nothing)
  const double lmax = fmaxf(key[0], 0.f);
  const double floor_ = 1e-6 * lmax;
  double ex = 0, top = 0, rem = 0, sub = 0;
  for (int64_t c = tid; c < a.s; c += nt) {
    const double lv = fmax(static_cast<double>(key[c]), 0.0);
    const double e = (sqrt(lv) - 1.0) * (sqrt(lv) - 1.0);
    if (c < nc) {
      ex += lv - 1.0;
      top += e;
    } else if (lv > 1.0) {
      rem += e;
    } else if (lv > floor_ && lv < 1.0) {
      sub += e;
    }
  }
  ex = block_sum(ex, red);
  top = block_sum(top, red);
  rem = block_sum(rem, red);
  sub = block_sum(sub, red);
  if (tid == 0) {
    const int mid = a.mat_ids[b];
    const float mprime = static_cast<float>(a.count[mid]);
    float* st = a.stats + 8 * b;
    st[0] = static_cast<float>(a.k_orient);
    st[1] = mprime;
    st[2] = fmaxf(mprime - static_cast<float>(ex), 0.f);
    st[3] = static_cast<float>(nc);
    st[4] = static_cast<float>(l);
    st[5] = static_cast<float>(a.n_a);
    st[6] = static_cast<float>(a.m_a);
    // outer sweeps that rotated a pair
    int sweeps = 0;
    for (int sw = 0; sw < kOjMaxSweeps; ++sw) sweeps += a.flag[sw * a.batch + b] != 0;
    st[7] = static_cast<float>(sweeps);
    if (a.diag) {
      double* d = a.diag + 8 * static_cast<int64_t>(mid);
      d[0] = top;
      d[1] = rem;
      d[2] = sub;
      d[3] = top + rem + sub;
    }
    if (a.flag[a.sweeps_flag_row * a.batch + b] != 0) raise_flag(a.flags, kFlagNumeric);   // no convergence
    if (!isfinite(lmax)) raise_flag(a.flags, kFlagNonfinite);
  }
}

// The selected eigenvectors: Q = z_c / sigma_c (Gamma on Z's long side), or
// the panel P = z_c / lambda_c that the caller multiplies by Psi_a.
struct OjVecArgs {
  const float* z; int64_t s_pad, lp;
  const int* sel; const float* sel_lam; int64_t sel_bs;
  float* out; int64_t out_bs;        // [n][l] row-major
  int64_t n;
  int l;
  int divide_by_lambda;              // 1: z / lambda; 0: z / sqrt(lambda)
};
__global__ void __launch_bounds__(256) k_oj_vectors(const __grid_constant__ OjVecArgs a) {
  const int b = blockIdx.y;
  const int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (e >= a.n * a.l) return;
  const int64_t i = e / a.l;
  const int c = static_cast<int>(e - i * a.l);
  const int col = a.sel[b * a.sel_bs + c];
  float v = 0.f;
  if (col >= 0) {
    const float lam = a.sel_lam[b * a.sel_bs + c];
    const float zv = a.z[(static_cast<int64_t>(b) * a.s_pad + col) * a.lp + i];
    v = a.divide_by_lambda ? zv / lam : zv * rsqrtf(lam);
  }
  a.out[b * a.out_bs + e] = v;
}

}  // namespace

cudaError_t exact_group_alloc(SketchGroup& g, std::vector<void*>& allocs) {
  const int64_t s = std::min(g.rows, g.cols), L = std::max(g.rows, g.cols);
  g.oj_s_pad = round_up(s, kOjP);
  g.oj_lp = round_up(L, kOjRows);
  auto alloc = [&](void** p, size_t bytes) -> cudaError_t {
    cudaError_t e = cudaMalloc(p, bytes);
    if (e == cudaSuccess) { allocs.push_back(*p); cudaMemset(*p, 0, bytes); }
    return e;
  };
  cudaError_t e;
  if ((e = alloc(reinterpret_cast<void**>(&g.oj_z), sizeof(float) * g.batch * g.oj_s_pad * g.oj_lp))) return e;
  if ((e = alloc(reinterpret_cast<void**>(&g.oj_lam), sizeof(float) * g.batch * g.oj_s_pad))) return e;
  if ((e = alloc(reinterpret_cast<void**>(&g.oj_flag), sizeof(int) * (kOjMaxSweeps + 1) * g.batch))) return e;
  if ((e = alloc(reinterpret_cast<void**>(&g.oj_sel), sizeof(int) * g.batch * g.lmax))) return e;
  if ((e = alloc(reinterpret_cast<void**>(&g.oj_sel_lam), sizeof(float) * g.batch * g.lmax))) return e;
  if ((e = alloc(reinterpret_cast<void**>(&g.eig_all), sizeof(float) * L * g.batch))) return e;
  cudaFuncSetAttribute(k_oj_round, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kOjSmem));
  // the largest selection any group can need (16384 eigenvalues and their
  // columns), so that every group's launch fits whichever group set it last
  cudaFuncSetAttribute(k_oj_select, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       static_cast<int>(kOjSelectMax * (sizeof(float) + sizeof(int))));
  return cudaGetLastError();
}

cudaError_t exact_eigs(SketchGroup& g, const SketchParams& p, int l, const int* mat_ids, const int* count,
                       double* diag, int* flags, cudaStream_t s, ProfileHook* prof, bool* needs_projection) {
  ProfileHook none;
  if (!prof) prof = &none;
  const bool rows_active = (p.k == 0);
  const int64_t m_a = rows_active ? g.rows : g.cols, n_a = rows_active ? g.cols : g.rows;
  const int64_t S = std::min(g.rows, g.cols), L = std::max(g.rows, g.cols);
  const int64_t big = L;
  const int64_t vbs = big * g.lmax;
  const int64_t sq = static_cast<int64_t>(g.lmax) * g.lmax;
  const int B = g.batch;
  cudaError_t e;
  prof->begin(kProfExactSweeps, s);
  {
    OjLoadArgs la;
    la.psi = g.psi; la.psi_bs = g.rows * g.ld; la.ld = g.ld;
    la.z = g.oj_z; la.s = S; la.s_pad = g.oj_s_pad; la.L = L; la.lp = g.oj_lp;
    la.cols_are_rows = g.rows <= g.cols;
    const dim3 grid(static_cast<unsigned>(cdiv(g.oj_lp, 32)), static_cast<unsigned>(cdiv(g.oj_s_pad, 32)), B);
    k_oj_load<<<grid, 256, 0, s>>>(la);
    if ((e = cudaGetLastError())) return e;
  }
  if ((e = cudaMemsetAsync(g.oj_flag, 0, sizeof(int) * (kOjMaxSweeps + 1) * B, s))) return e;
  const int nb = static_cast<int>(g.oj_s_pad / kOjB);
  int launches = 1;
  for (int sw = 0; sw < kOjMaxSweeps; ++sw) {
    for (int r = 0; r < nb - 1; ++r) {
      OjRoundArgs ra;
      ra.z = g.oj_z; ra.s_pad = g.oj_s_pad; ra.lp = g.oj_lp;
      ra.nb = nb; ra.round = r; ra.sweep = sw;
      ra.flag = g.oj_flag; ra.batch = B;
      ra.count = count; ra.mat_ids = mat_ids; ra.s = S;
      k_oj_round<<<dim3(nb / 2, B), 256, kOjSmem, s>>>(ra);
      if ((e = cudaGetLastError())) return e;
      ++launches;
    }
  }
  prof->end(kProfExactSweeps, s, launches);
  prof->begin(kProfExactSelect, s);
  {
    OjNormArgs na;
    na.z = g.oj_z; na.s = S; na.s_pad = g.oj_s_pad; na.lp = g.oj_lp; na.lam = g.oj_lam;
    k_oj_norms<<<dim3(static_cast<unsigned>(cdiv(g.oj_s_pad, 8)), B), 256, 0, s>>>(na);
    if ((e = cudaGetLastError())) return e;
  }
  {
    OjSelectArgs sa;
    sa.lam = g.oj_lam; sa.s = S; sa.s_pad = g.oj_s_pad; sa.m_a = m_a; sa.n_a = n_a;
    int npow = 1;
    while (npow < g.oj_s_pad) npow <<= 1;
    sa.npow = npow;
    sa.l = l; sa.rank = p.rank; sa.k_orient = p.k;
    // a last sweep that still rotated: the iteration had not converged
    sa.flag = g.oj_flag; sa.sweeps_flag_row = kOjMaxSweeps - 1; sa.batch = B;
    sa.eig_all = g.eig_all; sa.eig_bs = big;
    sa.ritz = g.ritz; sa.ritz_bs = g.lmax;
    sa.z = g.zvec; sa.kmat = g.kmat; sa.sq = sq;
    sa.stats = g.stats;
    sa.sel = g.oj_sel; sa.sel_lam = g.oj_sel_lam; sa.sel_bs = g.lmax;
    sa.diag = diag; sa.mat_ids = mat_ids;
    sa.count = count;
    sa.flags = flags;
    k_oj_select<<<B, 1024, npow * (sizeof(float) + sizeof(int)), s>>>(sa);
    if ((e = cudaGetLastError())) return e;
  }
  {
    // Gamma's eigenvectors on Z's long side (m_a = L): Q = z / sigma; else the
    // panel z / lambda (n_a = L rows), which the caller multiplies by Psi_a
    const bool cols_are_rows = g.rows <= g.cols;
    const bool direct = cols_are_rows == !rows_active;   // Gamma = Z Z^T
    OjVecArgs va;
    va.z = g.oj_z; va.s_pad = g.oj_s_pad; va.lp = g.oj_lp;
    va.sel = g.oj_sel; va.sel_lam = g.oj_sel_lam; va.sel_bs = g.lmax;
    va.l = l;
    if (direct) {
      va.out = g.q; va.out_bs = vbs; va.n = m_a; va.divide_by_lambda = 0;
    } else {
      va.out = g.y0; va.out_bs = vbs; va.n = n_a; va.divide_by_lambda = 1;
    }
    k_oj_vectors<<<dim3(static_cast<unsigned>(cdiv(va.n * l, 256)), B), 256, 0, s>>>(va);
    if ((e = cudaGetLastError())) return e;
    *needs_projection = !direct;
  }
  prof->end(kProfExactSelect, s, 3);
  return cudaSuccess;
}

}  // namespace normpre
