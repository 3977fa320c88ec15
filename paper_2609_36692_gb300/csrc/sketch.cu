// NormPre-L: randomized interaction sketch and localized preconditioner
// (Algorithm 2 and Sec. 2.3 of the paper), fused with the consistent-RMS weight
// update (Sec. 3.1).
//
// In the active orientation (m_a x n_a) the sketch computes
//   l = min(m_a, r + o);  Y = Psi Omega;  p times Y <- Psi (Psi^T Y);
//   Q = qr(Y);  B = Q^T Psi;  Gamma_Q = B B^T;  (Z, Lam) = eig(Gamma_Q);
//   C = {i <= min(r, l) : lam_i > 1};  T = Psi + Q K B,
//   K = Z_C (Lam_C^{-1/2} - I) Z_C^T,
// which equals Psi + U_C (Lam_C^{-1/2} - I) U_C^T Psi with U = Q Z, because
// U_C^T Psi = Z_C^T B.  Psi stays in the stored layout; a row-active step
// contracts over stored columns ("row contract": out = Psi V) and a
// column-active step over stored rows ("column contract": out = Psi^T U).
//
// Kernels: Philox4x32-10 Omega; SIMT skinny contractions (l <= 64 columns);
// split Gram sums Y^T Y in fp32 chunks folded in fp64; CholeskyQR (three
// passes, the first shifted when the Gram matrix is numerically singular) with
// an fp64 Cholesky and triangular inverse; a parallel (round-robin) cyclic
// Jacobi eigensolver in fp64 with a sweep cap; and a fused apply that forms
// T = Psi + L R^T tile by tile and updates W in the same pass.
//
// ||T||_F^2 comes from the closed form ||Psi||_F^2 - sum_C (lam_i - 1)
// (= m' - sum_C (lam_i - 1) for unit rows), which holds for any orthonormal Q
// and exact Ritz pairs of Gamma_Q (Lemma 2 of the paper gives the exact-case
// version), so W can be written in the same pass that forms T.
#include <algorithm>
#include <type_traits>

#include "common.cuh"
#include "internal.h"

namespace normpre {

constexpr int kLmax = 64;        // largest supported sketch width l
constexpr int kGramRows = 64;    // rows per fp32 chunk of the split Gram sums

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon et al., SC'11) and the Gaussian test matrix Omega
// ---------------------------------------------------------------------------
__device__ __forceinline__ void philox4x32_10(uint32_t c[4], uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t lo0 = 0xD2511F53u * c[0], hi0 = __umulhi(0xD2511F53u, c[0]);
    const uint32_t lo1 = 0xCD9E8D57u * c[2], hi1 = __umulhi(0xCD9E8D57u, c[2]);
    const uint32_t n0 = hi1 ^ c[1] ^ k0, n2 = hi0 ^ c[3] ^ k1;
    c[0] = n0; c[1] = lo1; c[2] = n2; c[3] = lo0;
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
}
// odd multiple of 2^-24 in (0, 1): exact in fp32
__device__ __forceinline__ float philox_unit(uint32_t x) {
  return (static_cast<float>(x >> 9) + 0.5f) * 1.1920928955078125e-07f;
}

struct OmegaArgs {
  float* omega;          // [batch][n_a][l]
  int64_t bstride;
  int64_t n_a;
  int l;
  uint32_t key0, key1, t_lo, t_hi;
  const int* mat_id;     // [batch]
};
__global__ void k_omega(const __grid_constant__ OmegaArgs a) {
  const int b = blockIdx.y;
  const int64_t n = a.n_a * a.l;
  const int64_t blk = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (blk * 4 >= n) return;
  uint32_t c[4] = {static_cast<uint32_t>(blk), static_cast<uint32_t>(a.mat_id[b]), a.t_lo, a.t_hi};
  philox4x32_10(c, a.key0, a.key1);
  float z[4];
#pragma unroll
  for (int p = 0; p < 2; ++p) {
    const float ua = philox_unit(c[2 * p]), ub = philox_unit(c[2 * p + 1]);
    const float rad = sqrtf(-2.f * logf(ua));
    float sn, cs;
    sincospif(2.f * ub, &sn, &cs);
    z[2 * p] = rad * cs;
    z[2 * p + 1] = rad * sn;
  }
  float* o = a.omega + b * a.bstride;
#pragma unroll
  for (int w = 0; w < 4; ++w)
    if (blk * 4 + w < n) o[blk * 4 + w] = z[w];
}

// ---------------------------------------------------------------------------
// Skinny contractions: out[P x l] = op(Psi) V,  op(Psi) = Psi (TRANS = false,
// P = rows, K = cols) or Psi^T (TRANS = true, P = cols, K = rows).
// V is [K x l] row-major (stride l), out is [P x l] (stride l).
// 64 x 64 output tiles, K chunks of 32, 256 threads x (4 x 4).
// ---------------------------------------------------------------------------
struct ContractArgs {
  const float* psi; int64_t psi_bs, psi_ld;
  const float* v; int64_t v_bs;
  float* out; int64_t out_bs;
  int64_t rows, cols;
  int l;
};
template <bool TRANS>
__global__ void __launch_bounds__(256) k_contract(const __grid_constant__ ContractArgs a) {
  __shared__ float Ps[32][64 + 4];
  __shared__ float Vs[32][64];
  const int b = blockIdx.y;
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
  const int64_t P = TRANS ? a.cols : a.rows, K = TRANS ? a.rows : a.cols;
  const int64_t p0 = static_cast<int64_t>(blockIdx.x) * 64;
  const float* psi = a.psi + b * a.psi_bs;
  const float* v = a.v + b * a.v_bs;
  const int l = a.l;
  float acc[4][4] = {};
  for (int64_t k0 = 0; k0 < K; k0 += 32) {
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const int e = tid + 256 * q;
      int i, k;
      if (TRANS) { k = e >> 6; i = e & 63; } else { i = e >> 5; k = e & 31; }
      const int64_t gp = p0 + i, gk = k0 + k;
      float x = 0.f;
      if (gp < P && gk < K) x = TRANS ? psi[gk * a.psi_ld + gp] : psi[gp * a.psi_ld + gk];
      Ps[k][i] = x;
    }
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const int e = tid + 256 * q;
      const int k = e >> 6, j = e & 63;
      const int64_t gk = k0 + k;
      Vs[k][j] = (j < l && gk < K) ? v[gk * l + j] : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int k = 0; k < 32; ++k) {
      float pv[4], vv[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) { pv[r] = Ps[k][ty * 4 + r]; vv[r] = Vs[k][tx * 4 + r]; }
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(pv[r], vv[c], acc[r][c]);
    }
    __syncthreads();
  }
  float* out = a.out + b * a.out_bs;
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int64_t gp = p0 + ty * 4 + r;
    if (gp >= P) continue;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int j = tx * 4 + c;
      if (j < l) out[gp * l + j] = acc[r][c];
    }
  }
}

// ---------------------------------------------------------------------------
// Split Gram sums: part[b][s] = sum over rows of chunk s of y_i y_i^T (fp64),
// each chunk accumulated in fp32 over kGramRows rows.  Y is [N x l].
// ---------------------------------------------------------------------------
struct GramArgs {
  const float* y; int64_t y_bs;
  double* part; int64_t part_bs;  // [nsplit][l][l] per matrix
  int64_t n;
  int l;
  int nsplit;
};
__global__ void __launch_bounds__(256) k_gram_part(const __grid_constant__ GramArgs a) {
  __shared__ float ys[kGramRows][kLmax];
  const int b = blockIdx.y, s = blockIdx.x, l = a.l;
  const int64_t i0 = static_cast<int64_t>(s) * kGramRows;
  const float* y = a.y + b * a.y_bs;
  for (int e = threadIdx.x; e < kGramRows * l; e += blockDim.x) {
    const int i = e / l, j = e - i * l;
    ys[i][j] = (i0 + i < a.n) ? y[(i0 + i) * l + j] : 0.f;
  }
  __syncthreads();
  double* out = a.part + b * a.part_bs + static_cast<int64_t>(s) * l * l;
  for (int e = threadIdx.x; e < l * l; e += blockDim.x) {
    const int p = e / l, q = e - p * l;
    float acc = 0.f;
    for (int i = 0; i < kGramRows; ++i) acc = fmaf(ys[i][p], ys[i][q], acc);
    out[e] = static_cast<double>(acc);
  }
}

// ---------------------------------------------------------------------------
// Small dense helpers on l x l matrices, one CTA per matrix.
// ---------------------------------------------------------------------------
struct CholArgs {
  const double* part; int64_t part_bs; int nsplit;
  double* work; int64_t work_bs;   // [2][l][l]: G, then R^{-1}
  float* rinv; int64_t rinv_bs;    // [l][l] fp32 copy of R^{-1}
  int l;
  int allow_shift;
  int* flags;
};
// Sums the Gram partials, Cholesky-factors G = R^T R (upper R) with one
// optional diagonal shift on breakdown, and writes R^{-1}.
__global__ void __launch_bounds__(256) k_chol_inv(const __grid_constant__ CholArgs a) {
  extern __shared__ double dsm[];
  __shared__ int bad;
  __shared__ double tr;
  const int b = blockIdx.x, l = a.l, tid = threadIdx.x;
  const int ld = l + 1;
  double* Gm = dsm;              // [l][l+1]
  double* Rm = dsm + l * ld;     // [l][l+1]
#define G(i, j) Gm[(i) * ld + (j)]
#define Ri(i, j) Rm[(i) * ld + (j)]
  const double* part = a.part + b * a.part_bs;
  for (int e = tid; e < l * l; e += blockDim.x) {
    double s = 0;
    for (int k = 0; k < a.nsplit; ++k) s += part[static_cast<int64_t>(k) * l * l + e];
    G(e / l, e % l) = s;
  }
  __syncthreads();
  if (tid == 0) {
    double t = 0;
    for (int i = 0; i < l; ++i) t += G(i, i);
    tr = t;
  }
  __syncthreads();
  for (int attempt = 0; attempt < 2; ++attempt) {
    // working copy in Ri (upper triangle), shifted on the second attempt
    const double shift = attempt == 0 ? 0.0 : 1e-6 * tr;
    for (int e = tid; e < l * l; e += blockDim.x) {
      const int i = e / l, j = e % l;
      Ri(i, j) = (j >= i) ? G(i, j) + (i == j ? shift : 0.0) : 0.0;
    }
    if (tid == 0) bad = 0;
    __syncthreads();
    for (int k = 0; k < l; ++k) {
      if (tid == 0) {
        const double d = Ri(k, k);
        if (!(d > 1e-13 * tr) || !isfinite(d)) bad = 1;
        Ri(k, k) = sqrt(fmax(d, 1e-300));
      }
      __syncthreads();
      const double dk = Ri(k, k);
      for (int j = k + 1 + tid; j < l; j += blockDim.x) Ri(k, j) /= dk;
      __syncthreads();
      for (int e = tid; e < l * l; e += blockDim.x) {
        const int i = e / l, j = e % l;
        if (i > k && j >= i) Ri(i, j) -= Ri(k, i) * Ri(k, j);
      }
      __syncthreads();
    }
    if (!bad || !a.allow_shift) break;
    __syncthreads();
  }
  float* ro = a.rinv + b * a.rinv_bs;
  if (!(tr > 0)) {
    // Y = 0 (a zero normalized update): Q = 0, nothing is selected downstream
    for (int e = tid; e < l * l; e += blockDim.x) ro[e] = 0.f;
    return;
  }
  if (tid == 0 && bad) raise_flag(a.flags, kFlagNumeric);
  // R is in Ri (upper).  Invert column by column: R X = I, X upper.
  // Store R in G (upper) and build X in Ri.
  for (int e = tid; e < l * l; e += blockDim.x) {
    const int i = e / l, j = e % l;
    G(i, j) = (j >= i) ? Ri(i, j) : 0.0;
  }
  __syncthreads();
  for (int j = tid; j < l; j += blockDim.x) {
    // back substitution for column j of X (X[i][j] = 0 for i > j)
    for (int i = l - 1; i >= 0; --i) {
      if (i > j) { Ri(i, j) = 0.0; continue; }
      double s = (i == j) ? 1.0 : 0.0;
      for (int k = i + 1; k <= j; ++k) s -= G(i, k) * Ri(k, j);
      Ri(i, j) = s / G(i, i);
    }
  }
  __syncthreads();
  for (int e = tid; e < l * l; e += blockDim.x) ro[e] = static_cast<float>(Ri(e / l, e % l));
#undef G
#undef Ri
}

// out[N x l] = Y[N x l] * S[l x l] (S fp32 row-major), one thread per output
struct RowMulArgs {
  const float* y; int64_t y_bs;
  const float* s; int64_t s_bs;
  float* out; int64_t out_bs;
  int64_t n;
  int l;
};
__global__ void __launch_bounds__(256) k_rowmul(const __grid_constant__ RowMulArgs a) {
  __shared__ float S[kLmax * kLmax];
  const int b = blockIdx.y, l = a.l;
  const float* s = a.s + b * a.s_bs;
  for (int e = threadIdx.x; e < l * l; e += blockDim.x) S[e] = s[e];
  __syncthreads();
  const int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (e >= a.n * l) return;
  const int64_t i = e / l;
  const int j = static_cast<int>(e - i * l);
  const float* y = a.y + b * a.y_bs + i * l;
  float acc = 0.f;
  for (int k = 0; k < l; ++k) acc = fmaf(y[k], S[k * l + j], acc);
  a.out[b * a.out_bs + e] = acc;
}

// ---------------------------------------------------------------------------
// Jacobi eigensolver of Gamma_Q (fp64), selection and K.
// ---------------------------------------------------------------------------
struct EigArgs {
  const double* part; int64_t part_bs; int nsplit;   // Gram partials of B^T
  float* ritz; int64_t ritz_bs;      // [l]
  float* z; int64_t z_bs;            // [l][l]
  float* kmat; int64_t k_bs;         // [l][l]
  float* stats; int64_t stats_bs;    // [8]
  const int* count; const int* mat_id;
  int l, rank, k_orient;
  int64_t m_a, n_a;
  int max_sweeps;
  int* flags;
};
__global__ void __launch_bounds__(256) k_jacobi(const __grid_constant__ EigArgs a) {
  extern __shared__ double dsm[];
  __shared__ double cs[kLmax / 2], sn[kLmax / 2];
  __shared__ int pp[kLmax / 2], qq[kLmax / 2];
  __shared__ double red[32];
  __shared__ int order[kLmax];
  const int b = blockIdx.x, l = a.l, tid = threadIdx.x;
  const int n = (l + 1) & ~1;          // even number of "players" (one dummy if l is odd)
  const int ld = l + 1;
  double* Am = dsm;              // [l][l+1]
  double* Vm = dsm + l * ld;     // [l][l+1]
#define A(i, j) Am[(i) * ld + (j)]
#define V(i, j) Vm[(i) * ld + (j)]
  const double* part = a.part + b * a.part_bs;
  for (int e = tid; e < l * l; e += blockDim.x) {
    double s = 0;
    for (int k = 0; k < a.nsplit; ++k) s += part[static_cast<int64_t>(k) * l * l + e];
    A(e / l, e % l) = s;
    V(e / l, e % l) = (e / l == e % l) ? 1.0 : 0.0;
  }
  __syncthreads();
  // symmetrize (the two triangles are summed in the same order, but be exact)
  for (int e = tid; e < l * l; e += blockDim.x) {
    const int i = e / l, j = e % l;
    if (i < j) { const double v = 0.5 * (A(i, j) + A(j, i)); A(i, j) = v; A(j, i) = v; }
  }
  __syncthreads();
  double diag2 = 0;
  {
    double s = 0;
    for (int i = tid; i < l; i += blockDim.x) s += A(i, i) * A(i, i);
    diag2 = block_sum(s, red);
  }
  int sweep = 0;
  __syncthreads();
  for (; sweep < a.max_sweeps; ++sweep) {
    for (int step = 0; step < n - 1; ++step) {
      // round-robin pairing: position 0 fixed, the others rotate by `step`
      for (int k = tid; k < n / 2; k += blockDim.x) {
        const int pa = k, pb = n - 1 - k;
        const int p = pa == 0 ? 0 : 1 + (pa - 1 + step) % (n - 1);
        const int q = 1 + (pb - 1 + step) % (n - 1);
        int i = min(p, q), j = max(p, q);
        double c = 1.0, s = 0.0;
        if (j < l) {
          const double apq = A(i, j);
          if (apq != 0.0) {
            const double th = (A(j, j) - A(i, i)) / (2.0 * apq);
            const double t = (th >= 0 ? 1.0 : -1.0) / (fabs(th) + sqrt(th * th + 1.0));
            c = 1.0 / sqrt(t * t + 1.0);
            s = t * c;
          }
        } else {
          i = j = -1;
        }
        pp[k] = i; qq[k] = j; cs[k] = c; sn[k] = s;
      }
      __syncthreads();
      // columns: A <- A J, V <- V J
      for (int e = tid; e < (n / 2) * l; e += blockDim.x) {
        const int k = e / l, r = e % l;
        const int i = pp[k], j = qq[k];
        if (i < 0) continue;
        const double c = cs[k], s = sn[k];
        const double ai = A(r, i), aj = A(r, j);
        A(r, i) = c * ai - s * aj;
        A(r, j) = s * ai + c * aj;
        const double vi = V(r, i), vj = V(r, j);
        V(r, i) = c * vi - s * vj;
        V(r, j) = s * vi + c * vj;
      }
      __syncthreads();
      // rows: A <- J^T A
      for (int e = tid; e < (n / 2) * l; e += blockDim.x) {
        const int k = e / l, r = e % l;
        const int i = pp[k], j = qq[k];
        if (i < 0) continue;
        const double c = cs[k], s = sn[k];
        const double ai = A(i, r), aj = A(j, r);
        A(i, r) = c * ai - s * aj;
        A(j, r) = s * ai + c * aj;
      }
      __syncthreads();
    }
    double off = 0;
    for (int e = tid; e < l * l; e += blockDim.x) {
      const int i = e / l, j = e % l;
      if (i != j) off += A(i, j) * A(i, j);
    }
    off = block_sum(off, red);
    if (off <= 1e-30 * diag2 || off == 0.0) { ++sweep; break; }
  }
  if (tid == 0 && sweep >= a.max_sweeps) raise_flag(a.flags, kFlagNumeric);
  // sort eigenvalues descending, ties by lower index (stable)
  for (int i = tid; i < l; i += blockDim.x) {
    const double li = A(i, i);
    int pos = 0;
    for (int j = 0; j < l; ++j) {
      const double lj = A(j, j);
      if (lj > li || (lj == li && j < i)) ++pos;
    }
    order[pos] = i;
  }
  __syncthreads();
  const int rr = min(a.rank, l);
  float* ritz = a.ritz + b * a.ritz_bs;
  float* z = a.z + b * a.z_bs;
  for (int c = tid; c < l; c += blockDim.x) ritz[c] = static_cast<float>(A(order[c], order[c]));
  for (int e = tid; e < l * l; e += blockDim.x) {
    const int r = e / l, c = e % l;
    z[e] = static_cast<float>(V(r, order[c]));
  }
  // K = sum_{c in C} (lam_c^{-1/2} - 1) z_c z_c^T
  float* km = a.kmat + b * a.k_bs;
  for (int e = tid; e < l * l; e += blockDim.x) {
    const int r = e / l, s = e % l;
    double acc = 0;
    for (int c = 0; c < rr; ++c) {
      const double lam = A(order[c], order[c]);
      if (!(lam > 1.0)) break;       // descending: the first lam <= 1 ends C
      acc += (1.0 / sqrt(lam) - 1.0) * V(r, order[c]) * V(s, order[c]);
    }
    km[e] = static_cast<float>(acc);
  }
  if (tid == 0) {
    int nc = 0;
    double excess = 0;
    for (int c = 0; c < rr; ++c) {
      const double lam = A(order[c], order[c]);
      if (!(lam > 1.0)) break;
      ++nc;
      excess += lam - 1.0;
    }
    const double mprime = static_cast<double>(a.count[a.mat_id[b]]);
    float* st = a.stats + b * a.stats_bs;
    st[0] = static_cast<float>(a.k_orient);
    st[1] = static_cast<float>(mprime);
    st[2] = static_cast<float>(fmax(mprime - excess, 0.0));
    st[3] = static_cast<float>(nc);
    st[4] = static_cast<float>(l);
    st[5] = static_cast<float>(a.n_a);
    st[6] = static_cast<float>(a.m_a);
    st[7] = static_cast<float>(sweep);
  }
}
#undef A
#undef V

// ---------------------------------------------------------------------------
// Fused apply: T = Psi + Lm R^T (Lm [rows x l], R [cols x l]) and
// W <- (1 - lr wd) W - lr * target * sqrt(mn) / ||T||_F * T
// ---------------------------------------------------------------------------
struct LApplyArgs {
  const float* psi; int64_t psi_bs, psi_ld;
  const float* lm; int64_t lm_bs;
  const float* rm; int64_t rm_bs;
  const float* stats; int64_t stats_bs;
  void* W[kMaxBatch];
  int64_t rows, cols;
  int l;
  float lr, wd, target;
};
template <typename TW>
__global__ void __launch_bounds__(256) k_apply_l(const __grid_constant__ LApplyArgs a) {
  __shared__ float Ls[kLmax][64 + 4];   // [p][row]
  __shared__ float Rs[kLmax][64 + 4];   // [p][col]
  const int b = blockIdx.z;
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
  const int64_t r0 = static_cast<int64_t>(blockIdx.y) * 64, c0 = static_cast<int64_t>(blockIdx.x) * 64;
  const int l = a.l;
  const float* lm = a.lm + b * a.lm_bs;
  const float* rm = a.rm + b * a.rm_bs;
  for (int e = tid; e < 64 * l; e += 256) {
    const int i = e / l, p = e - i * l;
    Ls[p][i] = (r0 + i < a.rows) ? lm[(r0 + i) * l + p] : 0.f;
    Rs[p][i] = (c0 + i < a.cols) ? rm[(c0 + i) * l + p] : 0.f;
  }
  __syncthreads();
  float acc[4][4] = {};
  for (int p = 0; p < l; ++p) {
    float lv[4], rv[4];
#pragma unroll
    for (int r = 0; r < 4; ++r) { lv[r] = Ls[p][ty * 4 + r]; rv[r] = Rs[p][tx * 4 + r]; }
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(lv[r], rv[c], acc[r][c]);
  }
  const float* st = a.stats + b * a.stats_bs;
  const double nrm2 = st[2];
  const double mn = static_cast<double>(a.rows) * static_cast<double>(a.cols);
  const float scale = nrm2 > 0 ? static_cast<float>(a.target * sqrt(mn / nrm2)) : 0.f;
  const float cw = 1.f - a.lr * a.wd, ct = -a.lr * scale;
  const float* psi = a.psi + b * a.psi_bs;
  TW* W = static_cast<TW*>(a.W[b]);
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int64_t i = r0 + ty * 4 + r;
    if (i >= a.rows) continue;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int64_t j = c0 + tx * 4 + c;
      if (j >= a.cols) continue;
      const float t = psi[i * a.psi_ld + j] + acc[r][c];
      const float w = to_f32(W[i * a.cols + j]);
      W[i * a.cols + j] = from_f32<TW>(fmaf(cw, w, ct * t));
    }
  }
}

// ---------------------------------------------------------------------------
// host orchestration
// ---------------------------------------------------------------------------
cudaError_t sketch_group_alloc(SketchGroup& g, int rank, int oversample, std::vector<void*>& allocs) {
  g.ell_rows = static_cast<int>(std::min<int64_t>(g.rows, rank + oversample));
  g.ell_cols = static_cast<int>(std::min<int64_t>(g.cols, rank + oversample));
  g.lmax = std::max(g.ell_rows, g.ell_cols);
  const int64_t big = std::max(g.rows, g.cols);
  g.max_part = static_cast<int>(cdiv(big, kGramRows));
  auto alloc = [&](void** p, size_t bytes) -> cudaError_t {
    cudaError_t e = cudaMalloc(p, bytes);
    if (e == cudaSuccess) { allocs.push_back(*p); cudaMemset(*p, 0, bytes); }
    return e;
  };
  const size_t vec = static_cast<size_t>(g.batch) * big * g.lmax * sizeof(float);
  const size_t sq = static_cast<size_t>(g.batch) * g.lmax * g.lmax;
  cudaError_t e;
  if ((e = alloc((void**)&g.psi, static_cast<size_t>(g.batch) * g.rows * g.ld * sizeof(float)))) return e;
  float** vbufs[] = {&g.omega, &g.y0, &g.zt, &g.y, &g.q, &g.bt, &g.qk};
  for (float** v : vbufs)
    if ((e = alloc((void**)v, vec))) return e;
  if ((e = alloc((void**)&g.part, static_cast<size_t>(g.batch) * g.max_part * g.lmax * g.lmax * sizeof(double)))) return e;
  if ((e = alloc((void**)&g.small, sq * 2 * sizeof(double)))) return e;
  if ((e = alloc((void**)&g.kmat, sq * sizeof(float)))) return e;
  if ((e = alloc((void**)&g.ritz, static_cast<size_t>(g.batch) * g.lmax * sizeof(float)))) return e;
  if ((e = alloc((void**)&g.zvec, sq * sizeof(float)))) return e;
  if ((e = alloc((void**)&g.stats, static_cast<size_t>(g.batch) * 8 * sizeof(float)))) return e;
  return cudaSuccess;
}

cudaError_t run_sketch_group(SketchGroup& g, const SketchParams& p, const int* mat_ids,
                             const int* count, void* const* W, int* flags, cudaStream_t s,
                             ProfileHook* prof) {
  ProfileHook none;
  if (!prof) prof = &none;
  const bool rows_active = (p.k == 0);
  const int64_t m_a = rows_active ? g.rows : g.cols, n_a = rows_active ? g.cols : g.rows;
  const int l = rows_active ? g.ell_rows : g.ell_cols;
  const int64_t big = std::max(g.rows, g.cols);
  const int64_t vbs = big * g.lmax;            // per-matrix stride of the l-wide buffers
  const int64_t psi_bs = g.rows * g.ld;
  const int B = g.batch;
  cudaError_t e;
#define NP_CHECK() do { e = cudaGetLastError(); if (e != cudaSuccess) return e; } while (0)

  // Omega [n_a x l]
  {
    OmegaArgs o;
    o.omega = g.omega; o.bstride = vbs; o.n_a = n_a; o.l = l;
    o.key0 = static_cast<uint32_t>(p.seed); o.key1 = static_cast<uint32_t>(p.seed >> 32);
    o.t_lo = static_cast<uint32_t>(static_cast<uint64_t>(p.t)); o.t_hi = static_cast<uint32_t>(static_cast<uint64_t>(p.t) >> 32);
    o.mat_id = mat_ids;
    const int64_t blocks = cdiv(n_a * l, 4);
    prof->begin(kProfOmega, s);
    k_omega<<<dim3(static_cast<unsigned>(cdiv(blocks, 256)), B), 256, 0, s>>>(o);
    NP_CHECK();
    prof->end(kProfOmega, s, 1);
  }
  // out = Psi_a V  (contract over the active row length n_a) or Psi_a^T U
  auto contract_a = [&](const float* v, float* out) -> cudaError_t {
    prof->begin(kProfContract, s);
    ContractArgs c;
    c.psi = g.psi; c.psi_bs = psi_bs; c.psi_ld = g.ld;
    c.v = v; c.v_bs = vbs; c.out = out; c.out_bs = vbs;
    c.rows = g.rows; c.cols = g.cols; c.l = l;
    if (rows_active) k_contract<false><<<dim3(static_cast<unsigned>(cdiv(g.rows, 64)), B), 256, 0, s>>>(c);
    else k_contract<true><<<dim3(static_cast<unsigned>(cdiv(g.cols, 64)), B), 256, 0, s>>>(c);
    prof->end(kProfContract, s, 1);
    return cudaGetLastError();
  };
  auto contract_at = [&](const float* u, float* out) -> cudaError_t {
    prof->begin(kProfContract, s);
    ContractArgs c;
    c.psi = g.psi; c.psi_bs = psi_bs; c.psi_ld = g.ld;
    c.v = u; c.v_bs = vbs; c.out = out; c.out_bs = vbs;
    c.rows = g.rows; c.cols = g.cols; c.l = l;
    if (rows_active) k_contract<true><<<dim3(static_cast<unsigned>(cdiv(g.cols, 64)), B), 256, 0, s>>>(c);
    else k_contract<false><<<dim3(static_cast<unsigned>(cdiv(g.rows, 64)), B), 256, 0, s>>>(c);
    prof->end(kProfContract, s, 1);
    return cudaGetLastError();
  };
  auto gram = [&](const float* y, int64_t n) -> int {
    GramArgs ga;
    ga.y = y; ga.y_bs = vbs; ga.part = g.part;
    ga.part_bs = static_cast<int64_t>(g.max_part) * g.lmax * g.lmax;
    ga.n = n; ga.l = l;
    ga.nsplit = static_cast<int>(cdiv(n, kGramRows));
    k_gram_part<<<dim3(ga.nsplit, B), 256, 0, s>>>(ga);
    return ga.nsplit;
  };
  // Y0 = Psi_a Omega; p times Y <- Psi_a (Psi_a^T Y)
  if ((e = contract_a(g.omega, g.y0))) return e;
  float* ycur = g.y0;
  for (int it = 0; it < p.power_iters; ++it) {
    if ((e = contract_at(ycur, g.zt))) return e;
    if ((e = contract_a(g.zt, g.y))) return e;
    ycur = g.y;
  }
  // Q = qr(Y): three CholeskyQR passes (the first may shift)
  prof->begin(kProfQR, s);
  {
    const float* src = ycur;
    for (int pass = 0; pass < 3; ++pass) {
      const int ns = gram(src, m_a);
      NP_CHECK();
      CholArgs ca;
      ca.part = g.part; ca.part_bs = static_cast<int64_t>(g.max_part) * g.lmax * g.lmax; ca.nsplit = ns;
      ca.work = g.small; ca.work_bs = 2 * static_cast<int64_t>(g.lmax) * g.lmax;
      ca.rinv = g.kmat; ca.rinv_bs = static_cast<int64_t>(g.lmax) * g.lmax;
      ca.l = l; ca.allow_shift = 1; ca.flags = flags;
      k_chol_inv<<<B, 256, 2 * l * (l + 1) * sizeof(double), s>>>(ca);
      NP_CHECK();
      float* dst = (pass == 1) ? g.zt : g.q;   // y -> q -> zt -> q
      RowMulArgs rm;
      rm.y = src; rm.y_bs = vbs; rm.s = g.kmat; rm.s_bs = static_cast<int64_t>(g.lmax) * g.lmax;
      rm.out = dst; rm.out_bs = vbs; rm.n = m_a; rm.l = l;
      k_rowmul<<<dim3(static_cast<unsigned>(cdiv(m_a * l, 256)), B), 256, 0, s>>>(rm);
      NP_CHECK();
      src = dst;
    }
  }
  prof->end(kProfQR, s, 9);
  // B^T = Psi_a^T Q  [n_a x l];  Gamma_Q = B B^T
  if ((e = contract_at(g.q, g.bt))) return e;
  prof->begin(kProfEig, s);
  {
    const int ns = gram(g.bt, n_a);
    NP_CHECK();
    EigArgs ea;
    ea.part = g.part; ea.part_bs = static_cast<int64_t>(g.max_part) * g.lmax * g.lmax; ea.nsplit = ns;
    ea.ritz = g.ritz; ea.ritz_bs = g.lmax;
    ea.z = g.zvec; ea.z_bs = static_cast<int64_t>(g.lmax) * g.lmax;
    ea.kmat = g.kmat; ea.k_bs = static_cast<int64_t>(g.lmax) * g.lmax;
    ea.stats = g.stats; ea.stats_bs = 8;
    ea.count = count; ea.mat_id = mat_ids;
    ea.l = l; ea.rank = p.rank; ea.k_orient = p.k;
    ea.m_a = m_a; ea.n_a = n_a;
    ea.max_sweeps = 40;
    ea.flags = flags;
    k_jacobi<<<B, 256, 2 * l * (l + 1) * sizeof(double), s>>>(ea);
    NP_CHECK();
  }
  // QK = Q K  [m_a x l]
  {
    RowMulArgs rm;
    rm.y = g.q; rm.y_bs = vbs; rm.s = g.kmat; rm.s_bs = static_cast<int64_t>(g.lmax) * g.lmax;
    rm.out = g.qk; rm.out_bs = vbs; rm.n = m_a; rm.l = l;
    k_rowmul<<<dim3(static_cast<unsigned>(cdiv(m_a * l, 256)), B), 256, 0, s>>>(rm);
    NP_CHECK();
  }
  prof->end(kProfEig, s, 3);
  // T_s = Psi + Lm R^T with (Lm, R) = (QK, B^T) row-active or (B^T, QK) column-active,
  // in launches of at most kMaxBatch matrices (W pointers travel as kernel arguments)
  prof->begin(kProfApplyL, s);
  int n_apply = 0;
  for (int c0 = 0; c0 < B; c0 += kMaxBatch) {
    const int nb = std::min(kMaxBatch, B - c0);
    ++n_apply;
    LApplyArgs la;
    la.psi = g.psi + c0 * psi_bs; la.psi_bs = psi_bs; la.psi_ld = g.ld;
    la.lm = (rows_active ? g.qk : g.bt) + c0 * vbs; la.lm_bs = vbs;
    la.rm = (rows_active ? g.bt : g.qk) + c0 * vbs; la.rm_bs = vbs;
    la.stats = g.stats + c0 * 8; la.stats_bs = 8;
    for (int i = 0; i < nb; ++i) la.W[i] = W[c0 + i];
    la.rows = g.rows; la.cols = g.cols; la.l = l;
    la.lr = p.lr; la.wd = p.wd; la.target = p.target;
    const dim3 grid(static_cast<unsigned>(cdiv(g.cols, 64)), static_cast<unsigned>(cdiv(g.rows, 64)), nb);
    if (g.w_dtype == 0) k_apply_l<float><<<grid, 256, 0, s>>>(la);
    else k_apply_l<bf16><<<grid, 256, 0, s>>>(la);
    NP_CHECK();
  }
  prof->end(kProfApplyL, s, n_apply);
#undef NP_CHECK
  return cudaSuccess;
}

}  // namespace normpre
