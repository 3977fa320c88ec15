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
// GB300 notes.  FP64 runs at a small fraction of the FP32 rate on this part,
// so every l x l kernel (Gram folds, Cholesky, triangular solve, Jacobi)
// works in fp32; sums that fold many partial results use compensated
// (Kahan) addition.  The l <= 72 wide products (contractions with Psi, the
// projector apply) keep one output row per thread with its l accumulators in
// registers and read the small operand from shared memory by broadcast, so
// they are bound by FMA issue rather than by shared-memory bandwidth; K is
// split (deterministic fixed-order reduce) when a launch would not fill the
// GPU.
//
// ||T||_F^2 comes from the closed form ||Psi||_F^2 - sum_C (lam_i - 1)
// (= m' - sum_C (lam_i - 1) for unit rows), which holds for any orthonormal Q
// and exact Ritz pairs of Gamma_Q (Lemma 2 of the paper gives the exact-case
// version), so W can be written in the same pass that forms T.
#include <algorithm>
#include <cstring>
#include <string>
#include <type_traits>

#include "../../include/normpre.h"
#include "common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace normpre {

constexpr int kLmax = 72;        // largest supported sketch width l (r = 64 with o = 8)
constexpr int kGramRows = 128;   // rows per fp32 chunk of the split Gram sums
constexpr int kMaxKSplit = 8;    // split-K factor bound of the contractions

// Kahan-compensated accumulator
struct Kahan {
  float s = 0.f, c = 0.f;
  __device__ __forceinline__ void add(float x) {
    const float y = x - c;
    const float t = s + y;
    c = (t - s) - y;
    s = t;
  }
};

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
  const int* mat_id;     // [batch]; null: every matrix is mat_id0
  int mat_id0 = 0;
  uint32_t* words = nullptr;   // optional [batch][n_a][l]: the Philox word of each element
  float* uniforms = nullptr;   // optional [batch][n_a][l]: its uniform in (0, 1)
};
static_assert(sizeof(OmegaArgs) + 64 <= 4096, "kernel arguments beyond 4 KB");
__global__ void k_omega(const __grid_constant__ OmegaArgs a) {
  const int b = blockIdx.y;
  const int64_t n = a.n_a * a.l;
  const int64_t blk = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (blk * 4 >= n) return;
  const int mid = a.mat_id ? a.mat_id[b] : a.mat_id0;
  uint32_t c[4] = {static_cast<uint32_t>(blk), static_cast<uint32_t>(mid), a.t_lo, a.t_hi};
  philox4x32_10(c, a.key0, a.key1);
  if (a.words != nullptr || a.uniforms != nullptr) {
#pragma unroll
    for (int w = 0; w < 4; ++w)
      if (blk * 4 + w < n) {
        if (a.words) a.words[b * a.bstride + blk * 4 + w] = c[w];
        if (a.uniforms) a.uniforms[b * a.bstride + blk * 4 + w] = philox_unit(c[w]);
      }
  }
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
// cp.async helpers (a zero source size fills the destination with zeros)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool valid) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(d), "l"(src), "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async4(void* dst, const void* src, bool valid) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(d), "l"(src), "r"(valid ? 4 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

// ---------------------------------------------------------------------------
// Skinny contractions: out[P x l] = op(Psi) V,  op(Psi) = Psi (TRANS = false,
// P = rows, K = cols) or Psi^T (TRANS = true, P = cols, K = rows).
// V is [K x l] row-major (stride l).  With ksplit > 1 every split writes a
// partial [P x l] block and k_split_reduce folds them in a fixed order.
//
// At l = 40 a contraction does 80 flops per 4-byte element of Psi, so it is
// bound by fp32 FMA issue, not HBM; the tiling aims at an FMA-to-shared-load
// ratio that keeps the FMA pipe busy.  Tile: 256 output rows x l columns,
// K chunks of 32 in two cp.async stages, 128 threads.  Lane (rq, ct) =
// (lane / 4, lane % 4) of warp w owns the 8 rows 64 w + rq + 8 i (interleaved,
// so a quarter warp's 16-byte reads of a K-major Psi tile hit distinct banks)
// and the CPT = ceil(l / 4) columns CPT ct .. CPT ct + CPT - 1: 8 x CPT
// accumulators per thread, about 0.9 bytes of shared memory per FMA.
// ---------------------------------------------------------------------------
struct ContractArgs {
  const float* psi; int64_t psi_bs, psi_ld;
  const float* v; int64_t v_bs;
  float* out; int64_t out_bs;      // final [P][l] or partials [ksplit][P][l]
  int64_t rows, cols;
  int l;
  int ksplit;
  int64_t kchunk;                  // K range of one split (multiple of 32)
};
static_assert(sizeof(ContractArgs) + 64 <= 4096, "kernel arguments beyond 4 KB");
constexpr int kCtP = 256, kCtK = 32, kCtThreads = 128;
constexpr int kCtPsiLd = kCtK + 4;          // non-TRANS: Ps[p][k]
constexpr int kCtPtLd = kCtP + 4;           // TRANS: Pt[k][p]
constexpr int kCtVLd = kLmax + 4;           // Vs[k][c]
constexpr int kCtPsiFloats = (kCtP * kCtPsiLd > kCtK * kCtPtLd) ? kCtP * kCtPsiLd : kCtK * kCtPtLd;
constexpr int kCtStageFloats = kCtPsiFloats + kCtK * kCtVLd;
constexpr size_t kCtSmem = 2 * kCtStageFloats * sizeof(float);

template <bool TRANS, int CPT>
__global__ void __launch_bounds__(kCtThreads) k_contract(const __grid_constant__ ContractArgs a) {
  extern __shared__ float4 ct_smem4[];
  float* smem = reinterpret_cast<float*>(ct_smem4);
  const int b = blockIdx.y, split = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rq = lane >> 2, ct = lane & 3;
  const int rbase = 64 * warp + rq;           // rows rbase + 8 i
  const int cbase = CPT * ct;                 // columns cbase .. cbase + CPT - 1
  const int64_t P = TRANS ? a.cols : a.rows, K = TRANS ? a.rows : a.cols;
  const int64_t p0 = static_cast<int64_t>(blockIdx.x) * kCtP;
  const int64_t kbeg = static_cast<int64_t>(split) * a.kchunk;
  const int64_t kend = min(K, kbeg + a.kchunk);
  const float* psi = a.psi + b * a.psi_bs;
  const float* v = a.v + b * a.v_bs;
  const int l = a.l;
  const int64_t ld = a.psi_ld;
  const bool v16 = (l % 4) == 0;

  auto load_stage = [&](int st, int64_t k0) {
    float* S = smem + st * kCtStageFloats;
    float* Vs = S + kCtPsiFloats;
#pragma unroll 4
    for (int q = 0; q < 16; ++q) {
      const int e = tid + kCtThreads * q;
      if (!TRANS) {
        const int row = e >> 3, k4 = (e & 7) * 4;      // 256 rows x 8 float4
        const int64_t gp = p0 + row, gk = k0 + k4;
        const bool ok = gp < P && gk < kend && gk + 4 <= ld;
        cp_async16(S + row * kCtPsiLd + k4, ok ? psi + gp * ld + gk : psi, ok);
      } else {
        const int k = e >> 6, p4 = (e & 63) * 4;       // 32 rows x 64 float4
        const int64_t gk = k0 + k, gp = p0 + p4;
        const bool ok = gk < kend && gp + 4 <= ld;
        cp_async16(S + k * kCtPtLd + p4, ok ? psi + gk * ld + gp : psi, ok);
      }
    }
    // V chunk as Vs[k][c]: rows of l floats (columns l .. 4 CPT - 1 zero)
    if (v16) {
      const int per = CPT;                              // float4 per padded row
      for (int e = tid; e < kCtK * per; e += kCtThreads) {
        const int k = e / per, c4 = (e - k * per) * 4;
        const int64_t gk = k0 + k;
        const bool ok = c4 < l && gk < kend;
        cp_async16(Vs + k * kCtVLd + c4, ok ? v + gk * l + c4 : v, ok);
      }
    } else {
      for (int e = tid; e < kCtK * 4 * CPT; e += kCtThreads) {
        const int k = e / (4 * CPT), c = e - k * (4 * CPT);
        const int64_t gk = k0 + k;
        const bool ok = c < l && gk < kend;
        cp_async4(Vs + k * kCtVLd + c, ok ? v + gk * l + c : v, ok);
      }
    }
    cp_async_commit();
  };

  float acc[8][CPT];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int c = 0; c < CPT; ++c) acc[i][c] = 0.f;

  int st = 0;
  if (kbeg < kend) load_stage(0, kbeg);
  for (int64_t k0 = kbeg; k0 < kend; k0 += kCtK) {
    if (k0 + kCtK < kend) {
      load_stage(st ^ 1, k0 + kCtK);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const float* S = smem + st * kCtStageFloats;
    const float* Vs = S + kCtPsiFloats + cbase;
    if (!TRANS) {
#pragma unroll 2
      for (int kk = 0; kk < kCtK; kk += 4) {
        float4 av[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) av[i] = *reinterpret_cast<const float4*>(S + (rbase + 8 * i) * kCtPsiLd + kk);
#pragma unroll
        for (int k4 = 0; k4 < 4; ++k4) {
          float bv[CPT];
#pragma unroll
          for (int c = 0; c < CPT; ++c) bv[c] = Vs[(kk + k4) * kCtVLd + c];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const float x = k4 == 0 ? av[i].x : k4 == 1 ? av[i].y : k4 == 2 ? av[i].z : av[i].w;
#pragma unroll
            for (int c = 0; c < CPT; ++c) acc[i][c] = fmaf(x, bv[c], acc[i][c]);
          }
        }
      }
    } else {
#pragma unroll 4
      for (int k = 0; k < kCtK; ++k) {
        float x[8], bv[CPT];
#pragma unroll
        for (int i = 0; i < 8; ++i) x[i] = S[k * kCtPtLd + rbase + 8 * i];
#pragma unroll
        for (int c = 0; c < CPT; ++c) bv[c] = Vs[k * kCtVLd + c];
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
          for (int c = 0; c < CPT; ++c) acc[i][c] = fmaf(x[i], bv[c], acc[i][c]);
      }
    }
    __syncthreads();
    st ^= 1;
  }
  float* out = a.out + b * a.out_bs + static_cast<int64_t>(split) * P * l;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int64_t gp = p0 + rbase + 8 * i;
    if (gp >= P) continue;
#pragma unroll
    for (int c = 0; c < CPT; ++c) {
      const int j = cbase + c;
      if (j < l) out[gp * l + j] = acc[i][c];
    }
  }
}

// ---------------------------------------------------------------------------
// Tensor-core form of the same contraction (tcgen05, kind::tf32) with fp32
// accuracy from three products per K step: every fp32 operand x is split into
// hi = x rounded to TF32 and lo = x - hi (exact in fp32) rounded to TF32, and
// A V = Ahi Vhi + Ahi Vlo + Alo Vhi up to the dropped Alo Vlo term and the
// rounding of lo: below 2^-21 relative per product (fp32 FMA: 2^-24).
//
// Psi, the streamed operand, goes to the tensor core through tensor memory:
// TMA copies 32-deep K blocks into shared memory as they lie (Psi K-major:
// box 32 x 128; Psi^T: four boxes of 32 K rows x 32 elements), eight warps
// read each row of the 128-row A tile (a quarter warp reads eight rows of one
// 16-byte chunk, or one word of 32 consecutive elements: no bank conflicts),
// split it in registers and write hi and lo into TMEM with tcgen05.st (lane =
// row, one 32-bit column per K element), where the MMAs read A.  Only the
// small V operand ([K][l], MN-major) is split into shared memory: the TF32
// MMA takes K-major shared-memory operands only, so its split also transposes
// (hi and lo tiles in the K-major 128-byte-swizzle layout, row r, 16-byte
// chunk j at r * 128 + ((j ^ (r & 7)) * 16)), while the TMEM stores drain.
// (Splitting V once per contraction in a kernel of its own, or freeing the
// Psi copies before the MMAs through a second ring, measured slower.)
//
// A TF32 MMA of M = 128, K = 8 costs the same ~94 cycles for any N up to 128
// (measured), so the three products take two instructions per K step: the V
// hi and lo tiles lie one after the other (rows 0..63 and 64..127 of one
// operand), and Ahi [Vhi; Vlo] (N = 64 + np, np = l rounded up to 16) fills
// accumulator columns 0..63 with Ahi Vhi and 64.. with Ahi Vlo, then Alo Vhi
// (N = np) adds into columns 0..np-1.
//
// The kernel is persistent: one CTA per SM walks the units (matrix, K split,
// 128-row tile), carrying its rings and accumulators from one unit to the
// next.  Warp 0 issues the TMA copies into a 6-slot input ring, which the
// split warps (2-9) free as soon as they have read a slot, so the copies run
// ahead of the split by up to six blocks; warp 1 issues the MMAs, which free
// the 4 operand stages (V hi / lo tiles, A hi / lo TMEM columns).  The tensor
// core's fp32 accumulation is biased toward zero by up to an ulp per
// addition, which over thousands of K steps reaches 1e-4 relative; so every
// kCtcSeg blocks the MMAs switch to the other of two TMEM accumulators, and
// warps 10-13 (one per TMEM lane quarter), which do nothing else, drain the
// finished one into fp32 registers with round-to-nearest additions (bias
// bounded by ~32 additions, ~2e-6) and write each unit's result.  (Draining
// from split warps stalled the split for the MMAs' completion every segment;
// sixteen split warps with eight drain warps measured slower than eight and
// four.)
// ---------------------------------------------------------------------------
struct ContractTcArgs {
  CUtensorMap psi_map;    // {cols, rows, batch} fp32, 128-byte swizzle
  CUtensorMap v_map;      // {l, K, batch} fp32, box 32 x 32
  float* out; int64_t out_bs;
  int64_t P, K;
  int l, np;              // np = MMA N = l rounded up to 16 (<= 64)
  int64_t kchunk;         // K range of one split (multiple of 32)
  int ksplit, batch;      // K splits and matrices (the units are tiles x ksplit x batch)
  int* flags;
  int stall_first_copy;   // tests: CTA 0 does not issue its first copy (its waits then give up)
};
static_assert(sizeof(ContractTcArgs) + 64 <= 4096, "kernel arguments beyond 4 KB");
// Two rings.  The input ring holds the TMA copies of the Psi block and of the
// V block; the split warps free a slot as soon as they have read it, so the
// copies run up to kCtcIn blocks ahead of the split and the HBM latency is
// covered by the copies in flight.  The MMA stages hold the split V hi / lo
// tiles in shared memory and the split A hi / lo in TMEM; the MMAs free them.
constexpr int kCtcIn = 6;                            // input ring slots
constexpr int kCtcStages = 4;                        // MMA operand stages
constexpr int kCtcSeg = 4;                           // K blocks per accumulator segment
constexpr int kCtcA = 128 * 32 * 4;                  // one A tile (128 rows x 32 K): 16 KB
constexpr int kCtcV = 64 * 32 * 4;                   // one V tile (64 rows x 32 K): 8 KB
constexpr int kCtcInSlot = kCtcA + kCtcV;            // Psi copy, V copy: 24 KB
constexpr int kCtcStage = 2 * kCtcV;                 // V hi, V lo: 16 KB
constexpr int kCtcSplitWarps = 8;
constexpr int kCtcDrainWarps = 4;
constexpr int kCtcThreads = 64 + 32 * (kCtcSplitWarps + kCtcDrainWarps);   // TMA, MMA, split, drain
constexpr size_t kCtcSmem = 1024 + kCtcIn * kCtcInSlot + kCtcStages * kCtcStage + 512;
// TMEM columns: two 128-column accumulators, then per stage 32 columns of A
// hi and 32 of A lo
constexpr uint32_t kCtcTmemA = 256;
constexpr uint32_t kCtcTmemCols = 512;
static_assert(kCtcTmemA + 64 * kCtcStages <= kCtcTmemCols, "TMEM budget");

// The three-product split of an fp32 operand: hi = x with the low 13
// mantissa bits cleared (a TF32 value, so the MMA reads it exactly), lo =
// x - hi (exact in fp32, |lo| < 2^-10 |x|).  The MMA reads lo at TF32
// precision, whatever rounding it applies to the dropped bits, which costs at
// most 2^-10 |lo| < 2^-20 |x|; the dropped lo * lo term is below 2^-20 of the
// product as well.
__device__ __forceinline__ float tf32_hi(float x) { return __uint_as_float(__float_as_uint(x) & 0xFFFFE000u); }
__device__ __forceinline__ void split4(const float4 x, float4& h, float4& l) {
  h.x = tf32_hi(x.x); l.x = x.x - h.x;
  h.y = tf32_hi(x.y); l.y = x.y - h.y;
  h.z = tf32_hi(x.z); l.z = x.z - h.z;
  h.w = tf32_hi(x.w); l.w = x.w - h.w;
}
// byte offset of 16-byte chunk j of row r in a 128-byte-swizzled tile
__device__ __forceinline__ uint32_t sw128(int r, int j) { return static_cast<uint32_t>(r * 128 + ((j ^ (r & 7)) << 4)); }

// MN-major source box (32 K rows x 32 elements, swizzled, rows = K) ->
// K-major rows r0 + c (c = lane) of the hi / lo tiles, K chunks j0 .. j0 + NJ - 1.
template <int NJ>
__device__ __forceinline__ void split_transpose(const uint8_t* box, uint8_t* hi, uint8_t* lo, int r0, int lane, int j0) {
  const int c = lane, r = r0 + c;
#pragma unroll
  for (int jj = 0; jj < NJ; ++jj) {        // K chunk j = K rows 4 j .. 4 j + 3
    const int j = j0 + jj;
    float4 x;
    x.x = *reinterpret_cast<const float*>(box + sw128(4 * j + 0, c >> 2) + 4 * (c & 3));
    x.y = *reinterpret_cast<const float*>(box + sw128(4 * j + 1, c >> 2) + 4 * (c & 3));
    x.z = *reinterpret_cast<const float*>(box + sw128(4 * j + 2, c >> 2) + 4 * (c & 3));
    x.w = *reinterpret_cast<const float*>(box + sw128(4 * j + 3, c >> 2) + 4 * (c & 3));
    float4 h, l;
    split4(x, h, l);
    *reinterpret_cast<float4*>(hi + sw128(r, j)) = h;
    *reinterpret_cast<float4*>(lo + sw128(r, j)) = l;
  }
}
// 16 consecutive 32-bit TMEM columns of the warp's 32 lanes: thread i writes
// lane (base + i).
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const float* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
      "%14, %15, %16};" ::"r"(taddr),
      "f"(v[0]), "f"(v[1]), "f"(v[2]), "f"(v[3]), "f"(v[4]), "f"(v[5]), "f"(v[6]), "f"(v[7]), "f"(v[8]), "f"(v[9]),
      "f"(v[10]), "f"(v[11]), "f"(v[12]), "f"(v[13]), "f"(v[14]), "f"(v[15])
      : "memory");
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// D[tmem] (+)= A[tmem] * B[smem]^T, kind::tf32
__device__ __forceinline__ void mma_tf32_ta(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

template <bool TRANS>
__global__ void __launch_bounds__(kCtcThreads, 1) k_contract_tc(const __grid_constant__ ContractTcArgs a) {
  extern __shared__ uint8_t ctc_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(ctc_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kCtcIn * kCtcInSlot + kCtcStages * kCtcStage);
                                             // [kCtcIn] copies landed
  uint64_t* inempty = full + kCtcIn;         // [kCtcIn] split warps done reading the slot
  uint64_t* splitb = inempty + kCtcIn;       // [kCtcStages] split written
  uint64_t* empty = splitb + kCtcStages;     // [kCtcStages] MMAs done with the stage
  uint64_t* tfull = empty + kCtcStages;      // [2] accumulator segment complete
  uint64_t* tempty = tfull + 2;              // [2] accumulator drained
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint32_t* issued = reinterpret_cast<uint32_t*>(tmem_slot + 2);   // [kCtcIn] last parity + 1
  // input slot: A copy | V copy; MMA stage: V hi | V lo
  auto a_copy = [&](int i) { return smem + i * kCtcInSlot; };
  auto v_copy = [&](int i) { return smem + i * kCtcInSlot + kCtcA; };
  auto v_split = [&](int st) { return smem + kCtcIn * kCtcInSlot + st * kCtcStage; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nvb = a.np > 32 ? 2 : 1;
  // work units u = (matrix b, K split z, row tile p), matrix-major so that
  // consecutive units share the V operand in L2; each CTA takes every
  // gridDim.x-th unit and carries its ring and accumulators across units
  const int tiles = static_cast<int>((a.P + 127) / 128);
  const int units = tiles * a.ksplit * a.batch;
  auto unit_of = [&](int u, int& b, int& z, int64_t& p0, int64_t& kbeg, int& nk) {
    p0 = static_cast<int64_t>(u % tiles) * 128;
    z = (u / tiles) % a.ksplit;
    b = u / (tiles * a.ksplit);
    kbeg = static_cast<int64_t>(z) * a.kchunk;
    const int64_t kend = min(a.K, kbeg + a.kchunk);
    nk = kend > kbeg ? static_cast<int>((kend - kbeg + 31) / 32) : 0;
  };
  if (threadIdx.x == 0) {
    for (int i = 0; i < kCtcIn; ++i) {
      tc::mbar_init(&full[i], 1);
      tc::mbar_init(&inempty[i], kCtcSplitWarps);
      issued[i] = 0;
    }
    for (int st = 0; st < kCtcStages; ++st) {
      tc::mbar_init(&splitb[st], kCtcSplitWarps);
      tc::mbar_init(&empty[st], 1);
    }
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&tfull[i], 1);
      tc::mbar_init(&tempty[i], kCtcDrainWarps);
    }
    *abort_flag = 0;
    tc::fence_barrier_init();
    tc::prefetch_map(&a.psi_map);
    tc::prefetch_map(&a.v_map);
  }
  if (warp == 1) {
    tc::tmem_alloc(tmem_slot, kCtcTmemCols);
    tc::tmem_relinquish();
    tc::fence_before();
  }
  // with l <= 32 the split writes rows 0..31 of V hi and lo only; rows 32..63
  // enter the wide MMA and must read as zero
  if (nvb == 1)
    for (int st = 0; st < kCtcStages; ++st)
      for (int i = threadIdx.x; i < 2 * kCtcV / 16; i += blockDim.x)
        reinterpret_cast<float4*>(v_split(st))[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    bool ok = true;
    uint32_t it = 0;
    for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
      int b, z, nk;
      int64_t p0, kbeg;
      unit_of(u, b, z, p0, kbeg, nk);
      for (int kb = 0; kb < nk && ok; ++kb, ++it) {
        const int i = it % kCtcIn;
        const uint32_t ph = (it / kCtcIn) & 1;
        ok = __all_sync(0xffffffffu, tc::mbar_wait(&inempty[i], ph ^ 1u, abort_flag));
        if (!ok) break;
        if (lane == 0 && !(a.stall_first_copy && blockIdx.x == 0 && it == 0)) {
          tc::mbar_expect_tx(&full[i], static_cast<uint32_t>(kCtcA + nvb * 4096));
          issued[i] = ph + 1;
          const int k0 = static_cast<int>(kbeg) + 32 * kb, pr = static_cast<int>(p0);
          if (!TRANS) {
            tc::tma_load_3d(a_copy(i), &a.psi_map, &full[i], k0, pr, b);
          } else {
#pragma unroll
            for (int j = 0; j < 4; ++j) tc::tma_load_3d(a_copy(i) + j * 4096, &a.psi_map, &full[i], pr + 32 * j, k0, b);
          }
          for (int j = 0; j < nvb; ++j) tc::tma_load_3d(v_copy(i) + j * 4096, &a.v_map, &full[i], 32 * j, k0, b);
        }
        __syncwarp();
      }
    }
    if (!ok && lane == 0) { *abort_flag = 1; raise_flag(a.flags, kFlagTimeout); }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    const uint32_t idesc_w = tc::idesc_tf32(128, 64 + a.np, 0, 0);   // Ahi [Vhi; Vlo]
    const uint32_t idesc_n = tc::idesc_tf32(128, a.np, 0, 0);        // Alo Vhi
    bool ok = true;
    uint32_t it = 0, gseg = 0;   // stage counter; segment counter over all units
    for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
      int b, z, nk;
      int64_t p0, kbeg;
      unit_of(u, b, z, p0, kbeg, nk);
      for (int kb = 0; kb < nk && ok; ++kb, ++it) {
        const int st = it % kCtcStages;
        const uint32_t ph = (it / kCtcStages) & 1;
        const bool seg_first = (kb % kCtcSeg) == 0;
        const bool seg_last = (kb % kCtcSeg) == kCtcSeg - 1 || kb == nk - 1;
        const int acc = gseg & 1;
        if (seg_first) {
          // the accumulator's previous segment has been drained
          ok = __all_sync(0xffffffffu, tc::mbar_wait(&tempty[acc], ((gseg >> 1) & 1) ^ 1u, abort_flag));
          if (!ok) break;
          tc::fence_after();
        }
        ok = __all_sync(0xffffffffu, tc::mbar_wait(&splitb[st], ph, abort_flag));
        if (!ok) break;
        tc::fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(128 * acc);
        if (lane == 0) {
          const uint32_t ahi = tmem_base + kCtcTmemA + 64u * st, alo = ahi + 32u;
          const uint32_t vhi = tc::su32(v_split(st));   // V lo follows at row 64
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {       // K step of 8: 8 TMEM columns of A, 32 bytes of a V row
            const uint64_t dv = tc::sdesc(vhi + kk * 32, 16, 1024);
            mma_tf32_ta(d_tmem, ahi + 8 * kk, dv, idesc_w, (!seg_first || kk != 0) ? 1u : 0u);
            mma_tf32_ta(d_tmem, alo + 8 * kk, dv, idesc_n, 1u);
          }
          tc::mma_commit(&empty[st]);
          if (seg_last) tc::mma_commit(&tfull[acc]);
        }
        __syncwarp();
        if (seg_last) ++gseg;
      }
    }
    if (!ok && lane == 0) { *abort_flag = 1; raise_flag(a.flags, kFlagTimeout); }
  } else if (warp < 2 + kCtcSplitWarps) {
    // ---------------- split (warps 2..9) ----------------
    const int w = warp - 2;
    const int q = warp & 3;        // TMEM lane quarter this warp may access
    const int kh = w >> 2;         // half of each 32-deep K block this warp splits
    bool ok = true;
    uint32_t it = 0;
    for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
      int b, z, nk;
      int64_t p0, kbeg;
      unit_of(u, b, z, p0, kbeg, nk);
      for (int kb = 0; kb < nk && ok; ++kb, ++it) {
        const int st = it % kCtcStages;
        const uint32_t ph = (it / kCtcStages) & 1;
        const int in = it % kCtcIn;
        ok = __all_sync(0xffffffffu, tc::mbar_wait(&full[in], (it / kCtcIn) & 1, abort_flag));
        if (!ok) break;
        // the MMAs are done with this stage's TMEM columns and V tiles
        ok = __all_sync(0xffffffffu, tc::mbar_wait(&empty[st], ph ^ 1u, abort_flag));
        if (!ok) break;
        tc::fence_after();
        const uint8_t* ac = a_copy(in);
        const uint8_t* vc = v_copy(in);
        uint8_t* vs = v_split(st);
        // A row r = 32 q + lane (the warp's TMEM lane quarter), K half kh
        {
          const int r = 32 * q + lane;
          float x[16], hi[16], lo[16];
          if (!TRANS) {
#pragma unroll
            for (int cc = 0; cc < 4; ++cc) {
              const float4 v = *reinterpret_cast<const float4*>(ac + sw128(r, 4 * kh + cc));
              x[4 * cc] = v.x; x[4 * cc + 1] = v.y; x[4 * cc + 2] = v.z; x[4 * cc + 3] = v.w;
            }
          } else {
            const uint8_t* box = ac + q * 4096;   // elements 32 q .. 32 q + 31, K rows 0..31
#pragma unroll
            for (int e = 0; e < 16; ++e)
              x[e] = *reinterpret_cast<const float*>(box + sw128(16 * kh + e, lane >> 2) + 4 * (lane & 3));
          }
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            hi[e] = tf32_hi(x[e]);
            lo[e] = x[e] - hi[e];
          }
          const uint32_t ta = tmem_base + (static_cast<uint32_t>(32 * q) << 16) + kCtcTmemA + 64u * st + 16u * kh;
          tmem_st16(ta, hi);
          tmem_st16(ta + 32u, lo);
        }
        // V (box w / 4, chunk pair w % 4 of two boxes, or box 0, chunk w of
        // one) while the TMEM stores drain
        if (nvb == 2) split_transpose<2>(vc + (w >> 2) * 4096, vs, vs + kCtcV, 32 * (w >> 2), lane, 2 * (w & 3));
        else split_transpose<1>(vc, vs, vs + kCtcV, 0, lane, w);
        // every read of the input slot has returned: hand it back to the copies
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&inempty[in]);
        tmem_st_wait();
        // the MMAs read V through the async proxy and A from TMEM
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        tc::fence_before();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&splitb[st]);
      }
    }
    if (!ok && lane == 0) { *abort_flag = 1; raise_flag(a.flags, kFlagTimeout); }
  } else {
    // ---------------- accumulator drains and unit results (warps 10..13) ----------------
    const int q = warp & 3;        // TMEM lane quarter: rows 32 q .. 32 q + 31 of the unit
    float sum[64];
    bool ok = true;
    uint32_t gseg = 0;
    for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
      int b, z, nk;
      int64_t p0, kbeg;
      unit_of(u, b, z, p0, kbeg, nk);
#pragma unroll
      for (int j = 0; j < 64; ++j) sum[j] = 0.f;
      // segments of kCtcSeg K blocks, as the MMA warp closes them
      const int nseg = (nk + kCtcSeg - 1) / kCtcSeg;
      for (int sg = 0; sg < nseg && ok; ++sg, ++gseg) {
        const int acc = gseg & 1;
        ok = __all_sync(0xffffffffu, tc::mbar_wait(&tfull[acc], (gseg >> 1) & 1, abort_flag));
        if (!ok) break;
        tc::fence_after();
#pragma unroll
        for (int h = 0; h < 4; ++h) {
          if (16 * h < a.np) {
            // Ahi Vhi + Alo Vhi in columns 16 h.., Ahi Vlo in 64 + 16 h..
            uint32_t r[16], v[16];
            const uint32_t col = tmem_base + (static_cast<uint32_t>(32 * q) << 16) + static_cast<uint32_t>(128 * acc + 16 * h);
            tc::tmem_ld16(col, r);
            tc::tmem_ld16(col + 64u, v);
            tc::tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 16; ++j) sum[16 * h + j] += __uint_as_float(r[j]) + __uint_as_float(v[j]);
          }
        }
        tc::fence_before();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&tempty[acc]);
      }
      if (!ok) break;
      const int64_t row = p0 + 32 * q + lane;
      float* out = a.out + b * a.out_bs + static_cast<int64_t>(z) * a.P * a.l;
      if (row < a.P) {
#pragma unroll
        for (int j = 0; j < 64; ++j)
          if (j < a.l) out[row * a.l + j] = sum[j];
      }
    }
    if (!ok && lane == 0) { *abort_flag = 1; raise_flag(a.flags, kFlagTimeout); }
  }
  __syncthreads();
  if (threadIdx.x == 0 && *abort_flag) {
    // let every TMA copy still in flight land before the CTA exits
    volatile int never = 0;
    for (int i = 0; i < kCtcIn; ++i)
      if (issued[i]) tc::mbar_wait(&full[i], issued[i] - 1, &never);
  }
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::fence_after();
    tc::tmem_dealloc(tmem_base, kCtcTmemCols);
  }
}

struct SplitReduceArgs {
  const float* part; int64_t part_bs;   // [ksplit][n] per matrix
  float* out; int64_t out_bs;
  int64_t n;
  int ksplit;
};
__global__ void k_split_reduce(const __grid_constant__ SplitReduceArgs a) {
  const int b = blockIdx.y;
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= a.n) return;
  const float* p = a.part + b * a.part_bs + i;
  float s = 0.f;
  for (int k = 0; k < a.ksplit; ++k) s += p[k * a.n];
  a.out[b * a.out_bs + i] = s;
}

// ---------------------------------------------------------------------------
// Split Gram sums: part[b][s] = sum over the rows of chunk s of y_i y_i^T,
// fp32 over kGramRows rows.  Y is [N x l].
// ---------------------------------------------------------------------------
// The 4 x 4 tiles on or above the diagonal of an l4 x l4 tile grid, numbered
// row by row: tile t -> (tp, tq) with tp <= tq, and back.  A Gram sum is
// symmetric entry for entry (the product y_ip y_iq is the same float for (p, q)
// and (q, p), added in the same order), so the kernels below sum only these
// tiles and mirror them.
__device__ __forceinline__ void upper_tile(int t, int l4, int& tp, int& tq) {
  int r = 0;
  while (t >= l4 - r) { t -= l4 - r; ++r; }
  tp = r;
  tq = r + t;
}
__device__ __forceinline__ int upper_index(int tp, int tq, int l4) { return tp * l4 - tp * (tp - 1) / 2 + (tq - tp); }
// entry (p, q) of the l x l sum as (upper tile, position in it)
__device__ __forceinline__ void upper_entry(int p, int q, int l4, int& tile, int& k) {
  const int tp = p >> 2, tq = q >> 2;
  if (tp <= tq) { tile = upper_index(tp, tq, l4); k = 4 * (p & 3) + (q & 3); }
  else { tile = upper_index(tq, tp, l4); k = 4 * (q & 3) + (p & 3); }
}

struct GramArgs {
  const float* y; int64_t y_bs;
  float* part; int64_t part_bs;   // [nsplit][l][l] per matrix
  int64_t n;
  int l;
  int nsplit;
};
static_assert(sizeof(GramArgs) + 64 <= 4096, "kernel arguments beyond 4 KB");
// One CTA per chunk.  The chunk is staged in shared memory; each thread
// accumulates a 4 x 4 block of the l x l sum over its share of the rows in
// registers (two 16-byte shared loads per 16 FMAs); when the blocks do not
// fill the CTA the rows are split into 2 or 4 groups whose sums are added in
// a fixed order.
__global__ void __launch_bounds__(256) k_gram_part(const __grid_constant__ GramArgs a) {
  constexpr int LD = kLmax + 4;                  // 16-byte rows
  __shared__ __align__(16) float ys[kGramRows * LD];
  const int b = blockIdx.y, s = blockIdx.x, l = a.l, tid = threadIdx.x;
  const int l4 = (l + 3) >> 2, lp = 4 * l4;
  const int64_t i0 = static_cast<int64_t>(s) * kGramRows;
  const int64_t nval = (a.n - i0 < kGramRows ? a.n - i0 : static_cast<int64_t>(kGramRows)) * l;   // valid floats of the chunk
  const float* y = a.y + b * a.y_bs + i0 * l;    // the chunk's rows are contiguous
  if ((l & 3) == 0 && (reinterpret_cast<uintptr_t>(y) & 15) == 0) {
    for (int e4 = tid; e4 < kGramRows * l / 4; e4 += blockDim.x) {
      const int e = 4 * e4, i = e / l, j = e - i * l;   // l % 4 == 0: one row per float4
      const float4 v = e < nval ? __ldg(reinterpret_cast<const float4*>(y) + e4) : make_float4(0.f, 0.f, 0.f, 0.f);
      *reinterpret_cast<float4*>(ys + i * LD + j) = v;
    }
  } else {
    for (int e = tid; e < kGramRows * l; e += blockDim.x) {
      const int i = e / l, j = e - i * l;
      ys[i * LD + j] = e < nval ? __ldg(y + e) : 0.f;
    }
  }
  for (int e = tid; e < kGramRows * (lp - l); e += blockDim.x) {
    const int i = e / (lp - l), j = l + (e - i * (lp - l));
    ys[i * LD + j] = 0.f;
  }
  __syncthreads();
  const int tiles = l4 * (l4 + 1) / 2;           // on or above the diagonal
  const int groups = tiles <= 64 ? 4 : (tiles <= 128 ? 2 : 1);
  const int rows_g = kGramRows / groups;
  float* out = a.part + b * a.part_bs + static_cast<int64_t>(s) * l * l;
  float acc[4][4];
  int my_tile = -1, my_group = 0;
  for (int t = tid; t < tiles * groups; t += blockDim.x) {
    const int tile = t % tiles, g = t / tiles;
    int tp, tq;
    upper_tile(tile, l4, tp, tq);
    const int p0 = 4 * tp, q0 = 4 * tq;
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[r][c] = 0.f;
    const float* yb = ys + g * rows_g * LD;
#pragma unroll 4
    for (int i = 0; i < rows_g; ++i) {
      const float4 pv = *reinterpret_cast<const float4*>(yb + i * LD + p0);
      const float4 qv = *reinterpret_cast<const float4*>(yb + i * LD + q0);
      const float pa[4] = {pv.x, pv.y, pv.z, pv.w}, qa[4] = {qv.x, qv.y, qv.z, qv.w};
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(pa[r], qa[c], acc[r][c]);
    }
    if (groups == 1) {
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c)
          if (p0 + r < l && q0 + c < l) {
            out[(p0 + r) * l + q0 + c] = acc[r][c];
            out[(q0 + c) * l + p0 + r] = acc[r][c];
          }
    } else {
      my_tile = tile;     // one (tile, group) per thread when groups > 1
      my_group = g;
    }
  }
  if (groups == 1) return;
  __syncthreads();                                // every read of ys is done: reuse it
  if (my_tile >= 0) {
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) ys[(my_group * tiles + my_tile) * 16 + 4 * r + c] = acc[r][c];
  }
  __syncthreads();
  for (int e = tid; e < l * l; e += blockDim.x) {
    const int p = e / l, q = e - p * l;
    int tile, k;
    upper_entry(p, q, l4, tile, k);
    float v = 0.f;
    for (int g = 0; g < groups; ++g) v += ys[(g * tiles + tile) * 16 + k];
    out[e] = v;
  }
}

// Folds nsplit partial l x l sums into dst (shared, row stride ld), compensated.
// Loads are issued sixteen at a time so their latencies overlap.
__device__ __forceinline__ void fold_partials(const float* part, int nsplit, int l, float* dst, int ld) {
  const int64_t stride = static_cast<int64_t>(l) * l;
  for (int e = threadIdx.x; e < l * l; e += blockDim.x) {
    Kahan k;
    int s = 0;
    for (; s + 16 <= nsplit; s += 16) {
      float v[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) v[u] = __ldcg(part + (s + u) * stride + e);
#pragma unroll
      for (int u = 0; u < 16; ++u) k.add(v[u]);
    }
    for (; s + 8 <= nsplit; s += 8) {
      float v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = __ldcg(part + (s + u) * stride + e);
#pragma unroll
      for (int u = 0; u < 8; ++u) k.add(v[u]);
    }
    for (; s < nsplit; ++s) k.add(__ldcg(part + s * stride + e));
    dst[(e / l) * ld + (e % l)] = k.s;
  }
}

// The nsplit partial l x l sums of each matrix folded once (one thread per
// entry, fixed order, compensated) into gram [batch][sq]: the consumers then
// read one value per entry instead of each walking the partials.
struct GramFoldArgs {
  const float* part; int64_t part_bs; int nsplit;
  float* gram; int64_t gram_bs;
  int l;
};
__global__ void __launch_bounds__(256) k_gram_fold(const __grid_constant__ GramFoldArgs a) {
  const int b = blockIdx.y;
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= a.l * a.l) return;
  const float* part = a.part + b * a.part_bs;
  const int64_t stride = static_cast<int64_t>(a.l) * a.l;
  Kahan k;
  int s = 0;
  for (; s + 8 <= a.nsplit; s += 8) {
    float v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) v[u] = __ldcg(part + (s + u) * stride + e);
#pragma unroll
    for (int u = 0; u < 8; ++u) k.add(v[u]);
  }
  for (; s < a.nsplit; ++s) k.add(__ldcg(part + s * stride + e));
  a.gram[b * a.gram_bs + e] = k.s;
}

// ---------------------------------------------------------------------------
// One CholeskyQR pass: one CTA per matrix folds the Gram matrix G of Y and
// factors G = R^T R (upper R, fp32); then every CTA of the solve reads R and
// solves q R = y for 256 rows of Y, one row per thread.  A pivot below
// 1e-6 tr(G) means Y is numerically rank
// deficient there: the first pass retries with the diagonal shifted by
// 1e-5 tr(G); the later passes, whose input is already well conditioned
// wherever it is not rank deficient, drop that column instead (a zero
// column of q, no elimination with it), so the kept columns stay
// orthonormal and a dropped one adds a zero Ritz value.
// The factorization is right-looking over the whole CTA (one pivot per
// barrier, the trailing square updated by a 16 x 16 thread grid); the solve
// is column-oriented (x_k final, then every later x_j updated from row k of
// R), so its dependent chain is l steps long, not l^2 / 2.  (Repeating the
// factorization in every solve CTA cost 1344 factorizations a pass on the
// 56 Qwen3 MLP matrices of 6144 rows.)
// ---------------------------------------------------------------------------
struct CholQRArgs {
  const float* part; int64_t part_bs; int nsplit;
  const float* y; float* q; int64_t v_bs;    // [n][l] panels
  int64_t n;
  int l;
  int vec;       // l % 4 == 0 and 16-byte aligned rows: float4 row loads / stores
  int drop;      // 0: shifted retry on a small pivot (first pass); 1: drop its column
  int* flags;
  float* gram_out; int64_t gram_bs;   // optional: per solve CTA, the l x l Gram sum of its rows
};
static_assert(sizeof(CholQRArgs) + 64 <= 4096, "kernel arguments beyond 4 KB");
// Per matrix [R (LP x LP, strictly upper, rows scaled by 1 / R_ii) | 1 / R_ii
// (LP) | zero-panel flag]: the factorization of one CholeskyQR pass, made
// once per matrix by k_chol_factor and read by every CTA of k_chol_solve.
constexpr int kRfacStride = kLmax * kLmax + kLmax + 8;

// One CTA per matrix: fold the Gram partials of the panel, factor G (+ shift)
// = R^T R right-looking (one pivot per barrier), write R and 1 / R_ii.
constexpr int kCholThreads = 1024;   // the fold of the Gram partials is latency-bound: many loads in flight
template <int LP>
__global__ void __launch_bounds__(kCholThreads) k_chol_factor(const __grid_constant__ CholQRArgs a, float* rfac) {
  // G (row stride LP + 1) until the factorization ends
  __shared__ __align__(16) float GR[LP * (LP + 1)];
  __shared__ float Wm[LP][LP + 1];             // G + shift I, reduced in place
  __shared__ float rinv[LP];                   // 1 / R_jj (zero past l)
  __shared__ float tr;
  const int b = blockIdx.x, l = a.l, tid = threadIdx.x;
  float* out = rfac + static_cast<int64_t>(b) * kRfacStride;
  fold_partials(a.part + b * a.part_bs, a.nsplit, l, GR, LP + 1);
  __syncthreads();
  if (tid < 32) {
    float t = 0.f;
    for (int i = tid; i < l; i += 32) t += GR[i * (LP + 1) + i];
    t = warp_sum(t);
    if (tid == 0) tr = t;
  }
  __syncthreads();
  if (!(tr > 0.f)) {
    // Y = 0 (a zero normalized update): Q = 0, nothing is selected downstream
    if (tid == 0) out[LP * LP + LP] = 1.f;
    return;
  }
  // right-looking Cholesky: at pivot j, W[p][q] -= W[j][p] W[j][q] / W[j][j]
  // for p, q > j (the whole trailing square, so W stays symmetric); row j is
  // final from then on and R[j][i] = W[j][i] / sqrt(W[j][j])
  const int ty = tid >> 5, tx = tid & 31;
  const float small = 1e-6f * tr;
  bool bad = false;
  for (int attempt = 0; attempt < 2; ++attempt) {
    const float shift = attempt == 0 ? 0.f : 1e-5f * tr;
    for (int e = tid; e < l * l; e += kCholThreads) {
      const int i = e / l, j = e - i * l;
      Wm[i][j] = GR[i * (LP + 1) + j] + (i == j ? shift : 0.f);
    }
    __syncthreads();
    bad = false;
    for (int j = 0; j < l; ++j) {
      const float d = Wm[j][j];
      const bool tiny = !(d > small);
      if (tiny) bad = true;
      // a dropped column eliminates nothing
      const float dinv = (tiny && a.drop) ? 0.f : 1.f / fmaxf(d, 1e-30f * tr);
      for (int p = j + 1 + ty; p < l; p += 32) {
        const float wp = Wm[j][p] * dinv;
        for (int c = j + 1 + tx; c < l; c += 32) Wm[p][c] = fmaf(-wp, Wm[j][c], Wm[p][c]);
      }
      __syncthreads();
    }
    if (!bad || a.drop) break;     // every thread saw the same pivots
  }
  if (tid == 0 && bad && !a.drop) raise_flag(a.flags, kFlagNumeric);
  // W[i][i] is pivot i; a dropped column gets 1 / R_ii = 0 (and so a zero row of R)
  for (int i = tid; i < LP; i += kCholThreads) {
    const float d = (i < l) ? Wm[i][i] : 0.f;
    rinv[i] = (i >= l || (a.drop && !(d > small))) ? 0.f : 1.f / sqrtf(fmaxf(d, 1e-30f * tr));
  }
  __syncthreads();
  for (int e = tid; e < LP * LP; e += kCholThreads) {
    const int i = e / LP, j = e % LP;
    out[e] = (i < l && j < l && j > i) ? Wm[i][j] * rinv[i] : 0.f;
  }
  for (int i = tid; i < LP; i += kCholThreads) out[LP * LP + i] = rinv[i];
  if (tid == 0) out[LP * LP + LP] = 0.f;
}

// The rows of Q: q R = y, one row per thread, with R from k_chol_factor.
template <int LP>
__global__ void __launch_bounds__(256) k_chol_solve(const __grid_constant__ CholQRArgs a, const float* rfac) {
  __shared__ __align__(16) float GR[LP * LP];  // R strictly above the diagonal, 16-byte rows
  __shared__ float rinv[LP];
  const int b = blockIdx.y, l = a.l, tid = threadIdx.x;
  const float* in = rfac + static_cast<int64_t>(b) * kRfacStride;
  const bool zero = in[LP * LP + LP] != 0.f;
  const int64_t row = static_cast<int64_t>(blockIdx.x) * 256 + tid;
  const float* y = a.y + b * a.v_bs + row * l;
  float* q = a.q + b * a.v_bs + row * l;
  if (zero) {
    if (row < a.n)
      for (int j = 0; j < l; ++j) q[j] = 0.f;
    return;
  }
  for (int e = tid; e < LP * LP / 4; e += 256)
    reinterpret_cast<float4*>(GR)[e] = __ldg(reinterpret_cast<const float4*>(in) + e);
  for (int i = tid; i < LP; i += 256) rinv[i] = in[LP * LP + i];
  __syncthreads();
  if (row >= a.n) return;
  float x[LP];
  if (a.vec) {
#pragma unroll
    for (int j = 0; j < LP; j += 4) {
      float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
      if (j < l) v = *reinterpret_cast<const float4*>(y + j);
      x[j] = v.x; x[j + 1] = v.y; x[j + 2] = v.z; x[j + 3] = v.w;
    }
  } else {
#pragma unroll
    for (int j = 0; j < LP; ++j) x[j] = (j < l) ? y[j] : 0.f;
  }
  // q R = y: x_k = x_k / R_kk is final, then x_j -= x_k R_kj for j > k
#pragma unroll
  for (int k = 0; k < LP; ++k) {
    x[k] *= rinv[k];
#pragma unroll
    for (int j4 = ((k + 1) / 4) * 4; j4 < LP; j4 += 4) {
      const float4 r = *reinterpret_cast<const float4*>(&GR[k * LP + j4]);
      if (j4 + 0 > k) x[j4 + 0] = fmaf(-x[k], r.x, x[j4 + 0]);
      if (j4 + 1 > k) x[j4 + 1] = fmaf(-x[k], r.y, x[j4 + 1]);
      if (j4 + 2 > k) x[j4 + 2] = fmaf(-x[k], r.z, x[j4 + 2]);
      if (j4 + 3 > k) x[j4 + 3] = fmaf(-x[k], r.w, x[j4 + 3]);
    }
  }
  if (a.vec) {
#pragma unroll
    for (int j = 0; j < LP; j += 4)
      if (j < l) *reinterpret_cast<float4*>(q + j) = make_float4(x[j], x[j + 1], x[j + 2], x[j + 3]);
  } else {
#pragma unroll
    for (int j = 0; j < LP; ++j)
      if (j < l) q[j] = x[j];
  }
}

// The solve of a pass whose result feeds another pass also sums the Gram
// matrix of its 256 rows (the next factorization folds one partial per solve
// CTA): the rows go through shared memory, 4 x 4 blocks of the l x l sum in
// registers per thread, rows split into groups when the blocks do not fill
// the CTA (summed in a fixed order).
template <int LP>
__global__ void __launch_bounds__(256) k_chol_solve_gram(const __grid_constant__ CholQRArgs a, const float* rfac) {
  extern __shared__ float4 sg_smem4[];
  float* X = reinterpret_cast<float*>(sg_smem4);          // [256][LP + 4]
  constexpr int LDX = LP + 4;
  __shared__ __align__(16) float GR[LP * LP];
  __shared__ float rinv[LP];
  const int b = blockIdx.y, l = a.l, tid = threadIdx.x;
  const float* in = rfac + static_cast<int64_t>(b) * kRfacStride;
  const bool zero = in[LP * LP + LP] != 0.f;
  const int64_t row = static_cast<int64_t>(blockIdx.x) * 256 + tid;
  const float* y = a.y + b * a.v_bs + row * l;
  float* q = a.q + b * a.v_bs + row * l;
  float x[LP];
#pragma unroll
  for (int j = 0; j < LP; ++j) x[j] = 0.f;
  if (!zero) {
    for (int e = tid; e < LP * LP / 4; e += 256)
      reinterpret_cast<float4*>(GR)[e] = __ldg(reinterpret_cast<const float4*>(in) + e);
    for (int i = tid; i < LP; i += 256) rinv[i] = in[LP * LP + i];
  }
  __syncthreads();
  if (row < a.n && !zero) {
    if (a.vec) {
#pragma unroll
      for (int j = 0; j < LP; j += 4) {
        float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
        if (j < l) v = *reinterpret_cast<const float4*>(y + j);
        x[j] = v.x; x[j + 1] = v.y; x[j + 2] = v.z; x[j + 3] = v.w;
      }
    } else {
#pragma unroll
      for (int j = 0; j < LP; ++j) x[j] = (j < l) ? y[j] : 0.f;
    }
#pragma unroll
    for (int k = 0; k < LP; ++k) {
      x[k] *= rinv[k];
#pragma unroll
      for (int j4 = ((k + 1) / 4) * 4; j4 < LP; j4 += 4) {
        const float4 r = *reinterpret_cast<const float4*>(&GR[k * LP + j4]);
        if (j4 + 0 > k) x[j4 + 0] = fmaf(-x[k], r.x, x[j4 + 0]);
        if (j4 + 1 > k) x[j4 + 1] = fmaf(-x[k], r.y, x[j4 + 1]);
        if (j4 + 2 > k) x[j4 + 2] = fmaf(-x[k], r.z, x[j4 + 2]);
        if (j4 + 3 > k) x[j4 + 3] = fmaf(-x[k], r.w, x[j4 + 3]);
      }
    }
  }
  if (row < a.n) {
    if (a.vec) {
#pragma unroll
      for (int j = 0; j < LP; j += 4)
        if (j < l) *reinterpret_cast<float4*>(q + j) = make_float4(x[j], x[j + 1], x[j + 2], x[j + 3]);
    } else {
#pragma unroll
      for (int j = 0; j < LP; ++j)
        if (j < l) q[j] = x[j];
    }
  }
  // rows past n and columns past l are zero
#pragma unroll
  for (int j = 0; j < LP; j += 4)
    *reinterpret_cast<float4*>(X + tid * LDX + j) = make_float4(x[j], x[j + 1], x[j + 2], x[j + 3]);
  __syncthreads();
  constexpr int L4 = LP / 4, TILES = L4 * (L4 + 1) / 2;   // tiles on or above the diagonal
  constexpr int GROUPS = TILES <= 64 ? 4 : (TILES <= 128 ? 2 : 1);
  constexpr int ROWS_G = 256 / GROUPS;
  float* out = a.gram_out + b * a.gram_bs + static_cast<int64_t>(blockIdx.x) * l * l;
  float acc[4][4];
  int my_tile = -1, my_group = 0;
  for (int t = tid; t < TILES * GROUPS; t += 256) {
    const int tile = t % TILES, g = t / TILES;
    int tp, tq;
    upper_tile(tile, L4, tp, tq);
    const int p0 = 4 * tp, q0 = 4 * tq;
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[r][c] = 0.f;
    const float* xb = X + g * ROWS_G * LDX;
#pragma unroll 4
    for (int i = 0; i < ROWS_G; ++i) {
      const float4 pv = *reinterpret_cast<const float4*>(xb + i * LDX + p0);
      const float4 qv = *reinterpret_cast<const float4*>(xb + i * LDX + q0);
      const float pa[4] = {pv.x, pv.y, pv.z, pv.w}, qa[4] = {qv.x, qv.y, qv.z, qv.w};
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(pa[r], qa[c], acc[r][c]);
    }
    if (GROUPS == 1) {
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c)
          if (p0 + r < l && q0 + c < l) {
            out[(p0 + r) * l + q0 + c] = acc[r][c];
            out[(q0 + c) * l + p0 + r] = acc[r][c];
          }
    } else {
      my_tile = tile;
      my_group = g;
    }
  }
  if (GROUPS == 1) return;
  __syncthreads();                                // X is read: reuse it for the group sums
  if (my_tile >= 0) {
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) X[(my_group * TILES + my_tile) * 16 + 4 * r + c] = acc[r][c];
  }
  __syncthreads();
  for (int e = tid; e < l * l; e += 256) {
    const int p = e / l, qq = e - p * l;
    int tile, k;
    upper_entry(p, qq, L4, tile, k);
    float v = 0.f;
    for (int g = 0; g < GROUPS; ++g) v += X[(g * TILES + tile) * 16 + k];
    out[e] = v;
  }
}

// out[N x l] = Y[N x l] * S[l x l] (S fp32 row-major), one thread per output
struct RowMulArgs {
  const float* y; int64_t y_bs;
  const float* s; int64_t s_bs;
  float* out; int64_t out_bs;
  int64_t n;
  int l;
};
// One thread per (row, 8 consecutive columns): the row's entries are
// broadcast loads shared by its threads, S's rows 16-byte shared loads.
__global__ void __launch_bounds__(256) k_rowmul(const __grid_constant__ RowMulArgs a) {
  __shared__ __align__(16) float S[kLmax * (kLmax + 8)];
  const int b = blockIdx.y, l = a.l;
  const int lp = (l + 7) & ~7, ld = lp;          // S rows padded with zeros to 8 columns
  const float* s = a.s + b * a.s_bs;
  for (int e = threadIdx.x; e < l * lp; e += blockDim.x) {
    const int k = e / lp, j = e - k * lp;
    S[k * ld + j] = j < l ? s[k * l + j] : 0.f;
  }
  __syncthreads();
  const int cg = lp >> 3;                        // column groups per row
  const int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (t >= a.n * cg) return;
  const int64_t i = t / cg;
  const int j0 = 8 * static_cast<int>(t - i * cg);
  const float* y = a.y + b * a.y_bs + i * l;
  float acc[8] = {};
  for (int k = 0; k < l; ++k) {
    const float yk = __ldg(y + k);
    const float4 s0 = *reinterpret_cast<const float4*>(S + k * ld + j0);
    const float4 s1 = *reinterpret_cast<const float4*>(S + k * ld + j0 + 4);
    acc[0] = fmaf(yk, s0.x, acc[0]); acc[1] = fmaf(yk, s0.y, acc[1]);
    acc[2] = fmaf(yk, s0.z, acc[2]); acc[3] = fmaf(yk, s0.w, acc[3]);
    acc[4] = fmaf(yk, s1.x, acc[4]); acc[5] = fmaf(yk, s1.y, acc[5]);
    acc[6] = fmaf(yk, s1.z, acc[6]); acc[7] = fmaf(yk, s1.w, acc[7]);
  }
  float* o = a.out + b * a.out_bs + i * l + j0;
#pragma unroll
  for (int c = 0; c < 8; ++c)
    if (j0 + c < l) o[c] = acc[c];
}

// ---------------------------------------------------------------------------
// Parallel cyclic Jacobi (round-robin pairing) of Gamma_Q in fp32, then the
// descending sort, the selection C and K.  One CTA per matrix.  The thread
// that owns 2 x 2 block (k, k') of the n/2 x n/2 block grid keeps the players
// of pairs k and k' in registers (advanced every step), forms both pairs'
// rotations from the current copy of A itself (every owner of a pair forms
// the same rotation from the same values), writes J^T A J for its block (rows
// rotated by pair k, columns by pair k') into the other copy of A and rotates
// rows k', k' + n/2 of V in pair k's columns: one barrier per rotation step.
// When l is odd the matrices are padded with a zero row and column whose pair
// is never rotated.
// ---------------------------------------------------------------------------
constexpr size_t kJacSmem = 3 * static_cast<size_t>(kLmax) * (kLmax + 1) * sizeof(float);
struct EigArgs {
  const float* part; int64_t part_bs; int nsplit;   // Gram partials of B^T
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
static_assert(sizeof(EigArgs) + 64 <= 4096, "kernel arguments beyond 4 KB");
// threads of k_jacobi for width l: one per 2 x 2 block (two each past 1024 blocks)
constexpr int kJacBlocks = ((kLmax / 2) * (kLmax / 2) + 1023) / 1024;
inline int64_t jacobi_threads(int l) {
  const int64_t np = (l + 1) / 2;
  return std::min<int64_t>(1024, ((np * np + 31) / 32) * 32);
}
// the rotation (c, s) that annihilates a_ij: t = tan(theta) is the smaller
// root of t^2 + 2 t cot(2 theta) - 1 = 0, cot(2 theta) = (a_jj - a_ii) / (2 a_ij)
__device__ __forceinline__ void jac_rot(float aii, float ajj, float aij, bool pad, float& c, float& s) {
  // branch-free: both branches of the guard are evaluated, then selected
  const bool skip = pad || !(fabsf(aij) > 1e-30f);
  const float th = __fdividef(ajj - aii, 2.f * aij);
  const float w = fmaf(th, th, 1.f);
  const float t_far = __fdividef(0.5f, th);    // t -> 1 / (2 cot(2 theta))
  const float t_near = __fdividef(copysignf(1.f, th), fabsf(th) + w * rsqrtf(w));
  const float t = fabsf(th) > 1e15f ? t_far : t_near;
  const float cc = rsqrtf(fmaf(t, t, 1.f));
  c = skip ? 1.f : cc;
  s = skip ? 0.f : t * cc;
}
__global__ void __launch_bounds__(1024) k_jacobi(const __grid_constant__ EigArgs a) {
  extern __shared__ float4 jc_smem4[];
  float* dsm = reinterpret_cast<float*>(jc_smem4);
  __shared__ float red[32];
  __shared__ int order[kLmax];
  const int b = blockIdx.x, l = a.l, tid = threadIdx.x, nt = blockDim.x;
  const int n = (l + 1) & ~1;          // even number of players (one padding player if l is odd)
  const int npairs = n / 2;
  const int ld = n + 1;
  float* cur = dsm;                    // A [n][ld], two copies
  float* nxt = dsm + n * ld;
  float* Vm = dsm + 2 * n * ld;        // V [n][ld]
#define V(i, j) Vm[(i) * ld + (j)]
  fold_partials(a.part + b * a.part_bs, a.nsplit, l, cur, ld);
  for (int e = tid; e < n * n; e += nt) {
    const int i = e / n, j = e - (e / n) * n;
    if (i >= l || j >= l) cur[i * ld + j] = 0.f;
    V(i, j) = (i == j) ? 1.f : 0.f;
  }
  __syncthreads();
  // exact symmetry
  for (int e = tid; e < l * l; e += nt) {
    const int i = e / l, j = e % l;
    if (i < j) {
      const float v = 0.5f * (cur[i * ld + j] + cur[j * ld + i]);
      cur[i * ld + j] = v;
      cur[j * ld + i] = v;
    }
  }
  __syncthreads();
  float frob2;
  {
    float s = 0.f;
    for (int e = tid; e < l * l; e += nt) {
      const float v = cur[(e / l) * ld + e % l];
      s += v * v;
    }
    frob2 = block_sum(s, red);
  }
  // pair k plays (p, q) = (k or 0, n - 1 - k) at step 0; every step moves
  // each player but player 0 on by one place in 1 .. n - 1
  int bk[kJacBlocks], bk2[kJacBlocks];
  int pa[kJacBlocks], qa[kJacBlocks], pb[kJacBlocks], qb[kJacBlocks];
#pragma unroll
  for (int it = 0; it < kJacBlocks; ++it) {
    const int e = tid + nt * it;
    bk[it] = (e < npairs * npairs) ? e / npairs : -1;
    bk2[it] = (e < npairs * npairs) ? e % npairs : 0;
  }
  auto advance = [&](int& p, int& q, int k) {
    if (k != 0) p = (p == n - 1) ? 1 : p + 1;
    q = (q == n - 1) ? 1 : q + 1;
  };
  int sweep = 0;
  float off = frob2, prev = frob2;
  for (; sweep < a.max_sweeps; ++sweep) {
#pragma unroll
    for (int it = 0; it < kJacBlocks; ++it) {
      const int k = bk[it] < 0 ? 0 : bk[it], k2 = bk2[it];
      pa[it] = k; qa[it] = n - 1 - k;
      pb[it] = k2; qb[it] = n - 1 - k2;
    }
    for (int step = 0; step < n - 1; ++step) {
#pragma unroll
      for (int it = 0; it < kJacBlocks; ++it) {
        const int k = bk[it], k2 = bk2[it];
        if (k >= 0) {
          const int i = min(pa[it], qa[it]), j = max(pa[it], qa[it]);
          const int i2 = min(pb[it], qb[it]), j2 = max(pb[it], qb[it]);
          float c, s, c2, s2;
          jac_rot(cur[i * ld + i], cur[j * ld + j], cur[i * ld + j], j >= l, c, s);
          jac_rot(cur[i2 * ld + i2], cur[j2 * ld + j2], cur[i2 * ld + j2], j2 >= l, c2, s2);
          const float* ri = cur + i * ld;
          const float* rj = cur + j * ld;
          const float a00 = ri[i2], a01 = ri[j2], a10 = rj[i2], a11 = rj[j2];
          // columns i2, j2 (A J), then rows i, j (J^T A)
          const float u0 = c2 * a00 - s2 * a01, w0 = s2 * a00 + c2 * a01;
          const float u1 = c2 * a10 - s2 * a11, w1 = s2 * a10 + c2 * a11;
          float* ni = nxt + i * ld;
          float* nj = nxt + j * ld;
          ni[i2] = c * u0 - s * u1; nj[i2] = s * u0 + c * u1;
          ni[j2] = c * w0 - s * w1; nj[j2] = s * w0 + c * w1;
          // V <- V J: rows k2 and k2 + n/2, columns of pair k
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            float* vr = Vm + (k2 + h * npairs) * ld;
            const float vi = vr[i], vj = vr[j];
            vr[i] = c * vi - s * vj;
            vr[j] = s * vi + c * vj;
          }
          advance(pa[it], qa[it], k);
          advance(pb[it], qb[it], k2);
        }
      }
      __syncthreads();
      float* t = cur; cur = nxt; nxt = t;
    }
    float so = 0.f;
    for (int e = tid; e < l * l; e += nt) {
      const int i = e / l, j = e % l;
      if (i != j) so += cur[i * ld + j] * cur[i * ld + j];
    }
    prev = off;
    off = block_sum(so, red);
    // converged, or stalled at the fp32 rounding floor (~ l^2 (u ||A||)^2):
    // Jacobi converges quadratically, so a sweep that no longer halves the
    // off-diagonal mass once it is tiny has reached that floor
    if (off <= 1e-12f * frob2 || (off <= 1e-9f * frob2 && off > 0.5f * prev)) { ++sweep; break; }
  }
#define A(i, j) cur[(i) * ld + (j)]
  if (tid == 0 && sweep >= a.max_sweeps && off > 1e-8f * frob2) raise_flag(a.flags, kFlagNumeric);
  // sort eigenvalues descending, ties by lower index (stable)
  for (int i = tid; i < l; i += nt) {
    const float li = A(i, i);
    int pos = 0;
    for (int j = 0; j < l; ++j) {
      const float lj = A(j, j);
      if (lj > li || (lj == li && j < i)) ++pos;
    }
    order[pos] = i;
  }
  __syncthreads();
  const int rr = min(a.rank, l);
  float* ritz = a.ritz + b * a.ritz_bs;
  float* z = a.z + b * a.z_bs;
  for (int c = tid; c < l; c += nt) ritz[c] = A(order[c], order[c]);
  for (int e = tid; e < l * l; e += nt) {
    const int r = e / l, c = e % l;
    z[e] = V(r, order[c]);
  }
  // K = sum_{c in C} (lam_c^{-1/2} - 1) z_c z_c^T
  float* km = a.kmat + b * a.k_bs;
  for (int e = tid; e < l * l; e += nt) {
    const int r = e / l, s = e % l;
    float acc = 0.f;
    for (int c = 0; c < rr; ++c) {
      const float lam = A(order[c], order[c]);
      if (!(lam > 1.f)) break;       // descending: the first lam <= 1 ends C
      acc = fmaf(rsqrtf(lam) - 1.f, V(r, order[c]) * V(s, order[c]), acc);
    }
    km[e] = acc;
  }
  if (tid == 0) {
    int nc = 0;
    float excess = 0.f;
    for (int c = 0; c < rr; ++c) {
      const float lam = A(order[c], order[c]);
      if (!(lam > 1.f)) break;
      ++nc;
      excess += lam - 1.f;
    }
    const float mprime = static_cast<float>(a.count[a.mat_id[b]]);
    float* st = a.stats + b * a.stats_bs;
    st[0] = static_cast<float>(a.k_orient);
    st[1] = mprime;
    st[2] = fmaxf(mprime - excess, 0.f);
    st[3] = static_cast<float>(nc);
    st[4] = static_cast<float>(l);
    st[5] = static_cast<float>(a.n_a);
    st[6] = static_cast<float>(a.m_a);
    st[7] = static_cast<float>(sweep);
  }
#undef A
#undef V
}


// ---------------------------------------------------------------------------
// Fused apply: T = Psi + Lm R^T (Lm [rows x l], R [cols x l]) and
// W <- (1 - lr wd) W - lr * target * sqrt(mn) / ||T||_F * T
// 64 x 64 tiles, thread = 4 x 4 block of consecutive rows / columns.
// ---------------------------------------------------------------------------
struct LApplyArgs {
  const void* psi; int64_t psi_bs, psi_ld;   // fp32, or bf16 when psi_bf16 (strides in elements)
  int psi_bf16;
  const float* lm; int64_t lm_bs;
  const float* rm; int64_t rm_bs;
  const float* stats; int64_t stats_bs;
  void* W[kMaxBatch];
  int64_t rows, cols;
  int l;
  float lr, wd, target;
  // DIAG: the step's gradients and, per matrix, where <G, T>, ||G||^2 and
  // ||T||^2 accumulate (fp64 atomics: diagnostics, not bitwise reproducible)
  const void* G[kMaxBatch];
  int g_dtype;
  double* diag[kMaxBatch];
  int vec_panels;   // l % 4 == 0 and 16-byte aligned panel rows: float4 panel loads
};
template <typename TW, bool VEC, bool DIAG>
__global__ void __launch_bounds__(256) k_apply_l(const __grid_constant__ LApplyArgs a) {
  __shared__ __align__(16) float Ls[kLmax][64 + 4];   // [p][row]
  __shared__ __align__(16) float Rs[kLmax][64 + 4];   // [p][col]
  double dgt = 0, dgg = 0, dtt = 0;
  auto diag_add = [&](int64_t idx, float t) {
    if (DIAG) {
      const float g = a.g_dtype ? to_f32(static_cast<const bf16*>(a.G[blockIdx.z])[idx])
                                : static_cast<const float*>(a.G[blockIdx.z])[idx];
      dgt += static_cast<double>(g) * t;
      dgg += static_cast<double>(g) * g;
      dtt += static_cast<double>(t) * t;
    }
  };
  const int b = blockIdx.z;
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
  const int64_t r0 = static_cast<int64_t>(blockIdx.y) * 64, c0 = static_cast<int64_t>(blockIdx.x) * 64;
  const int l = a.l;
  const float* lm = a.lm + b * a.lm_bs;
  const float* rm = a.rm + b * a.rm_bs;
  {
    // the 64 rows of Lm and the 64 of Rm, two threads per row (no division
    // by l: the load loop is a good part of the kernel's instructions)
    const int row = tid >> 1, half = tid & 1, i = row & 63;
    const bool right = row >= 64;
    const int64_t grow = (right ? c0 : r0) + i;
    const bool ok = grow < (right ? a.cols : a.rows);
    const float* src = (right ? rm : lm) + grow * l;
    float (*dst)[64 + 4] = right ? Rs : Ls;
    if (a.vec_panels) {
      // 16-byte pieces: q and q + 1 go to different halves of the bank space
      for (int q = half; q < (l >> 2); q += 2) {
        const float4 v = ok ? *reinterpret_cast<const float4*>(src + 4 * q) : make_float4(0.f, 0.f, 0.f, 0.f);
        dst[4 * q][i] = v.x;
        dst[4 * q + 1][i] = v.y;
        dst[4 * q + 2][i] = v.z;
        dst[4 * q + 3][i] = v.w;
      }
    } else {
      for (int p = half; p < l; p += 2) dst[p][i] = ok ? src[p] : 0.f;
    }
  }
  // the matrix's scale formed once (fp64 throughput is low on this part)
  __shared__ float scale_s;
  if (tid == 0) {
    const float nrm2 = a.stats[b * a.stats_bs + 2];
    const double mn = static_cast<double>(a.rows) * static_cast<double>(a.cols);
    scale_s = nrm2 > 0.f ? static_cast<float>(a.target * sqrt(mn / nrm2)) : 0.f;
  }
  __syncthreads();
  float acc[4][4] = {};
#pragma unroll 4
  for (int p = 0; p < l; ++p) {
    const float4 lv = *reinterpret_cast<const float4*>(&Ls[p][ty * 4]);
    const float4 rv = *reinterpret_cast<const float4*>(&Rs[p][tx * 4]);
    const float la[4] = {lv.x, lv.y, lv.z, lv.w}, ra[4] = {rv.x, rv.y, rv.z, rv.w};
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(la[r], ra[c], acc[r][c]);
  }
  const float cw = 1.f - a.lr * a.wd, ct = -a.lr * scale_s;
  const float* psi = static_cast<const float*>(a.psi) + b * a.psi_bs;
  const bf16* psib = static_cast<const bf16*>(a.psi) + b * a.psi_bs;
  TW* W = static_cast<TW*>(a.W[b]);
  const int64_t j0 = c0 + tx * 4;
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int64_t i = r0 + ty * 4 + r;
    if (i >= a.rows) continue;
    if (VEC && j0 + 4 <= a.cols) {
      float ps[4];
      if (a.psi_bf16) {
        const uint2 pv = *reinterpret_cast<const uint2*>(psib + i * a.psi_ld + j0);
        ps[0] = bf16lo(pv.x); ps[1] = bf16hi(pv.x); ps[2] = bf16lo(pv.y); ps[3] = bf16hi(pv.y);
      } else {
        const float4 pv = *reinterpret_cast<const float4*>(psi + i * a.psi_ld + j0);
        ps[0] = pv.x; ps[1] = pv.y; ps[2] = pv.z; ps[3] = pv.w;
      }
      float w[4];
      if (std::is_same<TW, float>::value) {
        const float4 wv = *reinterpret_cast<const float4*>(reinterpret_cast<float*>(W) + i * a.cols + j0);
        w[0] = wv.x; w[1] = wv.y; w[2] = wv.z; w[3] = wv.w;
      } else {
        const uint2 wv = *reinterpret_cast<const uint2*>(reinterpret_cast<bf16*>(W) + i * a.cols + j0);
        w[0] = bf16lo(wv.x); w[1] = bf16hi(wv.x); w[2] = bf16lo(wv.y); w[3] = bf16hi(wv.y);
      }
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        w[c] = fmaf(cw, w[c], ct * (ps[c] + acc[r][c]));
        diag_add(i * a.cols + j0 + c, ps[c] + acc[r][c]);
      }
      if (std::is_same<TW, float>::value) {
        *reinterpret_cast<float4*>(reinterpret_cast<float*>(W) + i * a.cols + j0) = make_float4(w[0], w[1], w[2], w[3]);
      } else {
        *reinterpret_cast<uint2*>(reinterpret_cast<bf16*>(W) + i * a.cols + j0) =
            make_uint2(pack_bf16x2(w[0], w[1]), pack_bf16x2(w[2], w[3]));
      }
    } else {
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int64_t j = j0 + c;
        if (j >= a.cols) continue;
        const float t = (a.psi_bf16 ? to_f32(psib[i * a.psi_ld + j]) : psi[i * a.psi_ld + j]) + acc[r][c];
        const float w = to_f32(W[i * a.cols + j]);
        W[i * a.cols + j] = from_f32<TW>(fmaf(cw, w, ct * t));
        diag_add(i * a.cols + j, t);
      }
    }
  }
  if (DIAG) {
    __shared__ double red[32];
    dgt = block_sum(dgt, red);
    dgg = block_sum(dgg, red);
    dtt = block_sum(dtt, red);
    if (threadIdx.x == 0) {
      atomicAdd(a.diag[b] + 4, dgt);
      atomicAdd(a.diag[b] + 5, dgg);
      atomicAdd(a.diag[b] + 6, dtt);
    }
  }
}

// ---------------------------------------------------------------------------
// Fused apply on the tensor cores (l % 4 == 0, l <= 64, no diagnostics).
// The rank-l product of T = Psi + Lm Rm^T runs as D = Rm_tile Lm_tile^T on
// tcgen05 kind::tf32 with the three-product split (hi hi + hi lo + lo hi, as
// the sketch contractions), M = 128 W columns and N = 256 W rows, so that the
// TMEM lane is the W column and the TMEM column the W row: an epilogue warp
// reading one TMEM column block then touches Psi and W in 128-byte rows
// across its 32 lanes, and the kernel is left with the compulsory HBM stream
// (Psi read, W read and write) instead of l fp32 FMAs per element.
//
// Persistent: CTA c takes a contiguous range of units (matrix, row tile,
// column tile), column tiles fastest, so the Lm tile is split once per row
// tile.  Warps 0-1 split the panel rows into the shared-memory operands
// (K-major, 128-byte swizzle, 32-wide K atoms), warp 2 issues the MMAs into
// one of two TMEM accumulators (256 columns each), warps 3-10 drain an
// accumulator into the weight update while the next unit's operands and MMAs
// proceed.
// ---------------------------------------------------------------------------
constexpr int kAtcRows = 256;                         // W rows per unit (MMA N)
constexpr int kAtcCols = 128;                         // W columns per unit (MMA M)
constexpr int kAtcProd = 2, kAtcEpi = 8;
constexpr int kAtcChunk = 16, kAtcSlots = 3;       // epilogue: rows per chunk, register ring slots
constexpr int kAtcThreads = 32 * (kAtcProd + 1 + kAtcEpi);
constexpr int kAtcAtomA = kAtcCols * 128;             // one 32-wide K atom of the A (Rm) tile
constexpr int kAtcAtomB = kAtcRows * 128;             // one 32-wide K atom of the B (Lm) tile
static size_t atc_smem(int natoms) { return 1024 + static_cast<size_t>(natoms) * 2 * (kAtcAtomA + kAtcAtomB) + 256; }

// rows [r0, r0 + R) of a panel (row stride l floats) split into hi / lo
// swizzled K-major tiles; rows past `nrows` are zero.  Eight 16-byte loads
// per thread are in flight before the first split.
template <int R>
__device__ __forceinline__ void atc_split_rows(const float* panel, int64_t r0, int64_t nrows, int l, uint8_t* hi,
                                               uint8_t* lo, int atom_bytes, int ptid) {
  constexpr int NT = 32 * kAtcProd, B = 8;
  const int l4 = l >> 2;
  const int n = R * l4;
  const float* src = panel + r0 * l;
  const int64_t valid = (nrows - r0) * l4;   // float4s of rows below nrows
  for (int base = ptid; base < n; base += B * NT) {
    float4 x[B];
#pragma unroll
    for (int k = 0; k < B; ++k) {
      const int idx = base + k * NT;
      x[k] = (idx < n && idx < valid) ? __ldg(reinterpret_cast<const float4*>(src) + idx)
                                      : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int k = 0; k < B; ++k) {
      const int idx = base + k * NT;
      if (idx < n) {
        const int r = idx / l4, c4 = idx - r * l4;
        float4 h, lw;
        split4(x[k], h, lw);
        const int kk = 4 * c4;
        const uint32_t off = static_cast<uint32_t>((kk >> 5) * atom_bytes) + sw128(r, (kk & 31) >> 2);
        *reinterpret_cast<float4*>(hi + off) = h;
        *reinterpret_cast<float4*>(lo + off) = lw;
      }
    }
  }
}

template <typename TW, typename TP>
__global__ void __launch_bounds__(kAtcThreads, 1) k_apply_tc(const __grid_constant__ LApplyArgs a, int nmat,
                                                              int natoms, int* flags) {
  extern __shared__ uint8_t atc_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(atc_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* a_hi = smem;
  uint8_t* a_lo = a_hi + natoms * kAtcAtomA;
  uint8_t* b_hi = a_lo + natoms * kAtcAtomA;
  uint8_t* b_lo = b_hi + natoms * kAtcAtomB;
  uint64_t* opfull = reinterpret_cast<uint64_t*>(b_lo + natoms * kAtcAtomB);   // operands written
  uint64_t* opfree = opfull + 1;                                               // MMAs done with them
  uint64_t* tfull = opfree + 1;                                                // [2] accumulator ready
  uint64_t* tempty = tfull + 2;                                                // [2] accumulator drained
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t rt = (a.rows + kAtcRows - 1) / kAtcRows, ct = (a.cols + kAtcCols - 1) / kAtcCols;
  const int64_t per_mat = rt * ct;
  const int64_t units = per_mat * nmat;
  const int64_t u0 = units * blockIdx.x / gridDim.x, u1 = units * (blockIdx.x + 1) / gridDim.x;
  // column tiles fastest: consecutive units of a CTA share the 256-row Lm tile
  auto unit_of = [&](int64_t u, int& b, int64_t& i0, int64_t& j0) {
    b = static_cast<int>(u / per_mat);
    const int64_t rem = u - b * per_mat;
    i0 = (rem / ct) * kAtcRows;
    j0 = (rem % ct) * kAtcCols;
  };
  if (threadIdx.x == 0) {
    tc::mbar_init(opfull, kAtcProd);
    tc::mbar_init(opfree, 1);
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&tfull[i], 1);
      tc::mbar_init(&tempty[i], kAtcEpi);
    }
    *abort_flag = 0;
    tc::fence_barrier_init();
  }
  if (warp == kAtcProd) {
    tc::tmem_alloc(tmem_slot, 512);
    tc::tmem_relinquish();
    tc::fence_before();
  }
  // K columns past l up to the next multiple of 8 enter the last MMA K step
  // and are never written below: zero the operand tiles once
  for (int i = threadIdx.x; i < natoms * 2 * (kAtcAtomA + kAtcAtomB) / 16; i += blockDim.x)
    reinterpret_cast<float4*>(smem)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int l = a.l;
  const int ksteps = (l + 7) / 8;

  if (warp < kAtcProd) {
    // ---------------- operand split ----------------
    const int ptid = threadIdx.x;
    bool ok = true;
    int64_t b_key = -1;
    uint32_t it = 0;
    for (int64_t u = u0; u < u1 && ok; ++u, ++it) {
      int b;
      int64_t i0, j0;
      unit_of(u, b, i0, j0);
      ok = __all_sync(0xffffffffu, tc::mbar_wait(opfree, (it & 1) ^ 1u, abort_flag));
      if (!ok) break;
      // the warps of this role finish the previous unit's writes before any
      // of them overwrites a tile: the MMAs that read them are done (opfree)
      const int64_t key = static_cast<int64_t>(b) * rt + i0 / kAtcRows;
      if (key != b_key)
        atc_split_rows<kAtcRows>(a.lm + b * a.lm_bs, i0, a.rows, l, b_hi, b_lo, kAtcAtomB, ptid);
      b_key = key;
      atc_split_rows<kAtcCols>(a.rm + b * a.rm_bs, j0, a.cols, l, a_hi, a_lo, kAtcAtomA, ptid);
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(opfull);
    }
    if (!ok && lane == 0) { *abort_flag = 1; raise_flag(flags, kFlagTimeout); }
  } else if (warp == kAtcProd) {
    // ---------------- MMA issuer ----------------
    const uint32_t idesc = tc::idesc_tf32(kAtcCols, kAtcRows, 0, 0);
    bool ok = true;
    uint32_t it = 0;
    for (int64_t u = u0; u < u1 && ok; ++u, ++it) {
      const int acc = it & 1;
      ok = __all_sync(0xffffffffu, tc::mbar_wait(opfull, it & 1, abort_flag));
      if (!ok) break;
      ok = __all_sync(0xffffffffu, tc::mbar_wait(&tempty[acc], ((it >> 1) & 1) ^ 1u, abort_flag));
      if (!ok) break;
      tc::fence_after();
      if (lane == 0) {
        const uint32_t d = tmem_base + static_cast<uint32_t>(256 * acc);
        for (int kk = 0; kk < ksteps; ++kk) {
          const uint32_t off = static_cast<uint32_t>(kk & 3) * 32u;
          const uint32_t aa = static_cast<uint32_t>(kk >> 2) * kAtcAtomA + off;
          const uint32_t bb = static_cast<uint32_t>(kk >> 2) * kAtcAtomB + off;
          const uint64_t dah = tc::sdesc(tc::su32(a_hi) + aa, 16, 1024), dal = tc::sdesc(tc::su32(a_lo) + aa, 16, 1024);
          const uint64_t dbh = tc::sdesc(tc::su32(b_hi) + bb, 16, 1024), dbl = tc::sdesc(tc::su32(b_lo) + bb, 16, 1024);
          tc::mma_tf32(d, dah, dbh, idesc, kk > 0 ? 1u : 0u);
          tc::mma_tf32(d, dah, dbl, idesc, 1u);
          tc::mma_tf32(d, dal, dbh, idesc, 1u);
        }
        tc::mma_commit(opfree);
        tc::mma_commit(&tfull[acc]);
      }
      __syncwarp();
    }
    if (!ok && lane == 0) { *abort_flag = 1; raise_flag(flags, kFlagTimeout); }
  } else {
    // ---------------- epilogue: W <- (1 - lr wd) W - lr s (Psi + D) ----------------
    // A stream of 16-row chunks (8 per unit: W rows 128 h .. 128 h + 127 of
    // the tile, W columns 32 q + lane): the Psi and W loads of a chunk do not
    // depend on the accumulator, so they are issued kAtcSlots - 1 chunks ahead
    // into a register ring and stay in flight while earlier chunks wait for
    // their MMAs and are combined.
    const int e = warp - kAtcProd - 1;
    const int q = warp & 3;          // TMEM lane quarter = W columns 32 q .. 32 q + 31 of the tile
    const int h = e >> 2;            // W rows 128 h .. 128 h + 127 of the tile
    const double mn = static_cast<double>(a.rows) * static_cast<double>(a.cols);
    const float cw = 1.f - a.lr * a.wd;
    constexpr int CH = kAtcChunk, NCH = 128 / kAtcChunk, S = kAtcSlots;
    const int64_t nck = (u1 - u0) * NCH;
    // issue cursor: the unit (matrix b, row tile i0, column tile j0) and chunk
    int ib;
    int64_t ii0, ij0;
    unit_of(u0, ib, ii0, ij0);
    int icc = 0;
    int cur_b = -1;
    float cur_ct = 0.f;
    TP pv[S][CH];
    TW wv[S][CH];
    TW* wp[S];
    int nr[S];
    float ctt[S];
    auto issue = [&](int64_t k, TP* P, TW* Wv, TW*& wptr, int& nrows, float& ct) {
      if (k < nck) {
        const int64_t j = ij0 + 32 * q + lane;
        const int64_t r0 = ii0 + 128 * h + CH * icc;
        if (ib != cur_b) {
          // fp64 throughput is low on this part: one lane per warp forms the
          // scale of a new matrix and broadcasts it
          float scale = 0.f;
          if (lane == 0) {
            const float nrm2 = a.stats[ib * a.stats_bs + 2];
            scale = nrm2 > 0.f ? static_cast<float>(a.target * sqrt(mn / nrm2)) : 0.f;
          }
          cur_ct = -a.lr * __shfl_sync(0xffffffffu, scale, 0);
          cur_b = ib;
        }
        ct = cur_ct;
        const TP* pptr = static_cast<const TP*>(a.psi) + ib * a.psi_bs + r0 * a.psi_ld + j;
        wptr = static_cast<TW*>(a.W[ib]) + r0 * a.cols + j;
        nrows = (r0 < a.rows && j < a.cols) ? static_cast<int>(a.rows - r0 < CH ? a.rows - r0 : CH) : 0;
        if (nrows == CH) {
#pragma unroll
          for (int rr = 0; rr < CH; ++rr) {
            P[rr] = __ldcs(pptr + rr * a.psi_ld);
            Wv[rr] = wptr[rr * a.cols];
          }
        } else {
#pragma unroll
          for (int rr = 0; rr < CH; ++rr) {
            P[rr] = rr < nrows ? pptr[rr * a.psi_ld] : from_f32<TP>(0.f);
            Wv[rr] = rr < nrows ? wptr[rr * a.cols] : from_f32<TW>(0.f);
          }
        }
        if (++icc == NCH) {
          icc = 0;
          ij0 += kAtcCols;
          if (ij0 >= a.cols) {
            ij0 = 0;
            ii0 += kAtcRows;
            if (ii0 >= a.rows) { ii0 = 0; ++ib; }
          }
        }
      }
    };
#pragma unroll
    for (int sl = 0; sl < S; ++sl) issue(sl, pv[sl], wv[sl], wp[sl], nr[sl], ctt[sl]);
    bool ok = true;
    for (int64_t k0 = 0; k0 < nck && ok; k0 += S) {
#pragma unroll
      for (int sl = 0; sl < S; ++sl) {
        const int64_t k = k0 + sl;
        if (k >= nck) break;
        const int64_t it = k / NCH;            // unit of this chunk, counted from u0
        const int c = static_cast<int>(k - it * NCH);
        const int acc = static_cast<int>(it & 1);
        if (c == 0) {
          ok = __all_sync(0xffffffffu, tc::mbar_wait(&tfull[acc], static_cast<uint32_t>((it >> 1) & 1), abort_flag));
          if (!ok) break;
          tc::fence_after();
        }
        uint32_t v[CH];
        tc::tmem_ld16(tmem_base + (static_cast<uint32_t>(32 * q) << 16) + static_cast<uint32_t>(256 * acc + 128 * h + CH * c), v);
        tc::tmem_ld_wait();
        if (c == NCH - 1) {
          // the accumulator is read: the MMAs of unit it + 2 may overwrite it
          tc::fence_before();
          __syncwarp();
          if (lane == 0) tc::mbar_arrive(&tempty[acc]);
        }
        TW* W = wp[sl];
        if (nr[sl] == CH) {
#pragma unroll
          for (int rr = 0; rr < CH; ++rr)
            W[rr * a.cols] = from_f32<TW>(fmaf(cw, to_f32(wv[sl][rr]), ctt[sl] * (to_f32(pv[sl][rr]) + __uint_as_float(v[rr]))));
        } else {
#pragma unroll
          for (int rr = 0; rr < CH; ++rr)
            if (rr < nr[sl])
              W[rr * a.cols] = from_f32<TW>(fmaf(cw, to_f32(wv[sl][rr]), ctt[sl] * (to_f32(pv[sl][rr]) + __uint_as_float(v[rr]))));
        }
        issue(k + S, pv[sl], wv[sl], wp[sl], nr[sl], ctt[sl]);
      }
    }
    if (!ok && lane == 0) { *abort_flag = 1; raise_flag(flags, kFlagTimeout); }
  }
  __syncthreads();
  if (warp == kAtcProd) {
    __syncwarp();
    tc::fence_after();
    tc::tmem_dealloc(tmem_base, 512);
  }
}

// ---------------------------------------------------------------------------
// host orchestration
// ---------------------------------------------------------------------------
#define NP_FOR_LP(X) X(8) X(16) X(24) X(32) X(40) X(48) X(56) X(64) X(72)

template <bool TRANS>
static cudaError_t launch_contract(const ContractArgs& c, int batch, int cpt, cudaStream_t s) {
  const int64_t P = TRANS ? c.cols : c.rows;
  const dim3 grid(static_cast<unsigned>(cdiv(P, kCtP)), static_cast<unsigned>(batch),
                  static_cast<unsigned>(c.ksplit));
  switch (cpt) {
#define NP_CT(N) case N: k_contract<TRANS, N><<<grid, kCtThreads, kCtSmem, s>>>(c); break;
    NP_CT(1) NP_CT(2) NP_CT(3) NP_CT(4) NP_CT(5) NP_CT(6) NP_CT(7) NP_CT(8)
    NP_CT(9) NP_CT(10) NP_CT(11) NP_CT(12) NP_CT(13) NP_CT(14) NP_CT(15) NP_CT(16)
    NP_CT(17) NP_CT(18)
#undef NP_CT
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

template <bool TRANS>
static void contract_attrs() {
#define NP_CT(N) \
  cudaFuncSetAttribute(k_contract<TRANS, N>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kCtSmem));
  NP_CT(1) NP_CT(2) NP_CT(3) NP_CT(4) NP_CT(5) NP_CT(6) NP_CT(7) NP_CT(8)
  NP_CT(9) NP_CT(10) NP_CT(11) NP_CT(12) NP_CT(13) NP_CT(14) NP_CT(15) NP_CT(16)
  NP_CT(17) NP_CT(18)
#undef NP_CT
}

static cudaError_t launch_cholqr(const CholQRArgs& c, float* rfac, int batch, int lp, cudaStream_t s) {
  const dim3 grid(static_cast<unsigned>(cdiv(c.n, 256)), static_cast<unsigned>(batch));
  switch (lp) {
#define NP_CQ(N)                                                                                        \
  case N:                                                                                               \
    k_chol_factor<N><<<batch, kCholThreads, 0, s>>>(c, rfac);                                                    \
    if (c.gram_out) {                                                                                   \
      const size_t sm = sizeof(float) * 256 * (N + 4);                                                  \
      static bool attr = false;                                                                         \
      if (!attr) {                                                                                      \
        cudaFuncSetAttribute(k_chol_solve_gram<N>, cudaFuncAttributeMaxDynamicSharedMemorySize,         \
                             static_cast<int>(sm));                                                     \
        attr = true;                                                                                    \
      }                                                                                                 \
      k_chol_solve_gram<N><<<grid, 256, sm, s>>>(c, rfac);                                              \
    } else {                                                                                            \
      k_chol_solve<N><<<grid, 256, 0, s>>>(c, rfac);                                                    \
    }                                                                                                   \
    break;
    NP_FOR_LP(NP_CQ)
#undef NP_CQ
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

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
  if ((e = alloc((void**)&g.kpart, vec * kMaxKSplit))) return e;
  if ((e = alloc((void**)&g.part, static_cast<size_t>(g.batch) * g.max_part * g.lmax * g.lmax * sizeof(float)))) return e;
  if ((e = alloc((void**)&g.kmat, sq * sizeof(float)))) return e;
  if ((e = alloc((void**)&g.gram, sq * sizeof(float)))) return e;
  if ((e = alloc((void**)&g.ritz, static_cast<size_t>(g.batch) * g.lmax * sizeof(float)))) return e;
  if ((e = alloc((void**)&g.zvec, sq * sizeof(float)))) return e;
  if ((e = alloc((void**)&g.stats, static_cast<size_t>(g.batch) * 8 * sizeof(float)))) return e;
  if ((e = alloc((void**)&g.rfac, static_cast<size_t>(g.batch) * kRfacStride * sizeof(float)))) return e;
  contract_attrs<false>();
  contract_attrs<true>();
  // tensor-core contractions: Psi as a 3-D tensor {cols, rows, batch}; the
  // l-wide operands need 16-byte rows and matrix strides (checked per launch)
  {
    const uint64_t dims[3] = {static_cast<uint64_t>(g.cols), static_cast<uint64_t>(g.rows),
                              static_cast<uint64_t>(g.batch)};
    const uint64_t strides[2] = {static_cast<uint64_t>(g.ld) * 4, static_cast<uint64_t>(g.rows * g.ld) * 4};
    const uint32_t box_k[3] = {32, 128, 1}, box_mn[3] = {32, 32, 1};
    g.tc = (g.ld % 4 == 0) && g.lmax <= 64 &&
           driver_encode_tiled(&g.psi_map_k, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, g.psi, dims, strides, box_k, nullptr) &&
           driver_encode_tiled(&g.psi_map_mn, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, g.psi, dims, strides, box_mn, nullptr);
    if (g.tc) {
      cudaFuncSetAttribute(k_contract_tc<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kCtcSmem));
      cudaFuncSetAttribute(k_contract_tc<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kCtcSmem));
    }
  }
  // bf16 Psi (set by the caller for NORMPRE_L in NORMPRE_PREC_BF16): kept only
  // where the bf16 contraction applies (l <= 64, 16-byte Psi rows)
  if (g.psi_bf16) {
    g.vb_bs = 2 * round_up(g.lmax, 16) * round_up(big, 64);
    g.psi_bf16 = g.lmax <= 64 && contract_bf16_map(&g.psi_map_bf, g.psi, g.rows, g.cols, g.ld, g.batch) &&
                 contract_bf16_map(&g.psi_map_apply, g.psi, g.rows, g.cols, g.ld, g.batch, 32);
    if (g.psi_bf16 && (e = alloc(&g.vb, static_cast<size_t>(g.batch) * g.vb_bs * sizeof(uint16_t)))) return e;
  }
  // the largest Jacobi footprint, so that groups of any width can share the kernel
  cudaFuncSetAttribute(k_jacobi, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kJacSmem));
  return cudaGetLastError();
}

cudaError_t sketch_group_slice(const SketchGroup& g, int b0, int b1, SketchGroup* out) {
  if (b0 < 0 || b0 >= b1 || b1 > g.batch) return cudaErrorInvalidValue;
  SketchGroup s = g;
  const int64_t vbs = std::max(g.rows, g.cols) * g.lmax;
  const int64_t sq = static_cast<int64_t>(g.lmax) * g.lmax;
  s.batch = b1 - b0;
  s.plan_batch = g.plan_batch ? g.plan_batch : g.batch;
  s.psi = g.psi_bf16 ? reinterpret_cast<float*>(reinterpret_cast<uint16_t*>(g.psi) + b0 * g.rows * g.ld)
                     : g.psi + b0 * g.rows * g.ld;
  if (g.psi_bf16) {
    s.vb = static_cast<uint16_t*>(g.vb) + b0 * g.vb_bs;
    if (!contract_bf16_map(&s.psi_map_bf, s.psi, g.rows, g.cols, g.ld, s.batch) ||
        !contract_bf16_map(&s.psi_map_apply, s.psi, g.rows, g.cols, g.ld, s.batch, 32))
      return cudaErrorInvalidValue;
  }
  float** vbufs[] = {&s.omega, &s.y0, &s.zt, &s.y, &s.q, &s.bt, &s.qk};
  for (float** v : vbufs) *v += b0 * vbs;
  s.kpart = g.kpart + b0 * vbs * kMaxKSplit;
  s.part = g.part + b0 * static_cast<int64_t>(g.max_part) * sq;
  s.kmat = g.kmat + b0 * sq;
  s.gram = g.gram + b0 * sq;
  s.zvec = g.zvec + b0 * sq;
  s.ritz = g.ritz + static_cast<int64_t>(b0) * g.lmax;
  s.stats = g.stats + static_cast<int64_t>(b0) * 8;
  s.rfac = g.rfac + static_cast<int64_t>(b0) * kRfacStride;
  if (g.eig_all) s.eig_all = g.eig_all + b0 * std::max(g.rows, g.cols);
  if (g.oj_z) {
    s.oj_z = g.oj_z + b0 * g.oj_s_pad * g.oj_lp;
    s.oj_lam = g.oj_lam + b0 * g.oj_s_pad;
    s.oj_flag = g.oj_flag + b0 * static_cast<int64_t>(kExactFlagRows);
    s.oj_sel = g.oj_sel + static_cast<int64_t>(b0) * g.lmax;
    s.oj_sel_lam = g.oj_sel_lam + static_cast<int64_t>(b0) * g.lmax;
  }
  if (g.tc && !g.psi_bf16) {
    const uint64_t dims[3] = {static_cast<uint64_t>(g.cols), static_cast<uint64_t>(g.rows),
                              static_cast<uint64_t>(s.batch)};
    const uint64_t strides[2] = {static_cast<uint64_t>(g.ld) * 4, static_cast<uint64_t>(g.rows * g.ld) * 4};
    const uint32_t box_k[3] = {32, 128, 1}, box_mn[3] = {32, 32, 1};
    s.tc = driver_encode_tiled(&s.psi_map_k, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, s.psi, dims, strides, box_k, nullptr) &&
           driver_encode_tiled(&s.psi_map_mn, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, s.psi, dims, strides, box_mn, nullptr);
  }
  *out = s;
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
  const int lp = static_cast<int>(round_up(l, 8));   // register width of the QR solves
  const int cpt = (l + 3) / 4;                         // columns per thread of the contractions
  const int64_t sq = static_cast<int64_t>(g.lmax) * g.lmax;
  cudaError_t e;
#define NP_CHECK() do { e = cudaGetLastError(); if (e != cudaSuccess) return e; } while (0)

  // Omega [n_a x l] (the sketch only)
  if (!p.exact) {
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
  // out = op(Psi) V; op = Psi contracts over stored columns, Psi^T over stored
  // rows.  K is split when the tiles alone would leave SMs idle (fixed-order reduce).
  // the tensor-core form needs 16-byte rows of the l-wide operand and 16-byte
  // aligned per-matrix strides (TMA)
  const bool use_tc = g.psi_bf16 || (g.tc && (l % 4 == 0) && (vbs % 4 == 0) && l <= 64);
  bool stall_pending = p.test_stall != 0;   // the first tensor-core contraction of the step
  auto contract = [&](bool trans, const float* v, float* out) -> cudaError_t {
    prof->begin(kProfContract, s);
    const int64_t P = trans ? g.cols : g.rows, K = trans ? g.rows : g.cols;
    const int64_t tiles = cdiv(P, use_tc ? 128 : kCtP) * (g.plan_batch ? g.plan_batch : B);
    int ks = 1;
    const int64_t want = (use_tc ? 1 : 2) * static_cast<int64_t>(device_sm_count());
    while (ks < kMaxKSplit && tiles * ks < want && K / (2 * ks) >= 256) ks *= 2;
    ContractArgs c;
    c.psi = g.psi; c.psi_bs = psi_bs; c.psi_ld = g.ld;
    c.v = v; c.v_bs = vbs;
    c.rows = g.rows; c.cols = g.cols; c.l = l;
    c.ksplit = ks;
    c.kchunk = round_up(cdiv(K, ks), kCtK);
    if (ks == 1) {
      c.out = out; c.out_bs = vbs;
    } else {
      c.out = g.kpart; c.out_bs = vbs * kMaxKSplit;
    }
    cudaError_t err;
    if (g.psi_bf16) {
      ContractBf16Launch cb;
      cb.psi_map = &g.psi_map_bf; cb.trans = trans;
      cb.v = v; cb.v_bs = vbs;
      cb.vb = g.vb; cb.vb_bs = g.vb_bs;
      cb.out = c.out; cb.out_bs = c.out_bs;
      cb.P = P; cb.K = K; cb.l = l;
      cb.kchunk = round_up(cdiv(K, ks), 64);
      cb.ksplit = ks; cb.batch = B;
      cb.flags = flags;
      cb.stall_first_copy = stall_pending ? 1 : 0;
      stall_pending = false;
      err = launch_contract_bf16(cb, s);
    } else if (use_tc) {
      const int np = static_cast<int>(round_up(l, 16));
      ContractTcArgs ct;
      std::memset(static_cast<void*>(&ct), 0, sizeof(ct));
      ct.psi_map = trans ? g.psi_map_mn : g.psi_map_k;
      const uint64_t vdims[3] = {static_cast<uint64_t>(l), static_cast<uint64_t>(K), static_cast<uint64_t>(B)};
      const uint64_t vstr[2] = {static_cast<uint64_t>(l) * 4, static_cast<uint64_t>(vbs) * 4};
      const uint32_t vbox[3] = {32, 32, 1};
      std::string why;
      if (!driver_encode_tiled(&ct.v_map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<float*>(v), vdims, vstr,
                               vbox, &why))
        return cudaErrorInvalidValue;
      ct.out = c.out; ct.out_bs = c.out_bs;
      ct.P = P; ct.K = K; ct.l = l; ct.np = np;
      ct.kchunk = c.kchunk;
      ct.flags = flags;
      ct.ksplit = ks; ct.batch = B;
      ct.stall_first_copy = stall_pending ? 1 : 0;
      stall_pending = false;
      // persistent: one CTA per SM (shared memory and TMEM admit one)
      const int64_t units = cdiv(P, 128) * ks * B;
      const unsigned grid = static_cast<unsigned>(std::min<int64_t>(units, device_sm_count()));
      if (trans) k_contract_tc<true><<<grid, kCtcThreads, kCtcSmem, s>>>(ct);
      else k_contract_tc<false><<<grid, kCtcThreads, kCtcSmem, s>>>(ct);
      err = cudaGetLastError();
    } else {
      err = trans ? launch_contract<true>(c, B, cpt, s) : launch_contract<false>(c, B, cpt, s);
    }
    if (err) return err;
    int n_l = g.psi_bf16 ? 2 : 1;   // the bf16 path splits V in a launch of its own
    if (ks > 1) {
      SplitReduceArgs r;
      r.part = g.kpart; r.part_bs = vbs * kMaxKSplit;
      r.out = out; r.out_bs = vbs;
      r.n = P * l; r.ksplit = ks;
      k_split_reduce<<<dim3(static_cast<unsigned>(cdiv(r.n, 256)), B), 256, 0, s>>>(r);
      err = cudaGetLastError();
      if (err) return err;
      ++n_l;
    }
    prof->end(kProfContract, s, n_l);
    return cudaSuccess;
  };
  const bool ta = !rows_active;     // Psi_a V:   row contract (k = 0) or column contract (k = 1)
  const bool tb = rows_active;      // Psi_a^T U: the other one
  // Gram partials of an n x l panel, folded once per matrix into g.gram when
  // there is more than one; returns where the consumer reads them (pointer,
  // matrix stride, count of partial sums)
  struct GramOut { const float* p; int64_t bs; int n; };
  int n_fold = 0;   // fold launches (for the per-class launch counts)
  auto gram = [&](const float* y, int64_t n) -> GramOut {
    GramArgs ga;
    ga.y = y; ga.y_bs = vbs; ga.part = g.part;
    ga.part_bs = static_cast<int64_t>(g.max_part) * sq;
    ga.n = n; ga.l = l;
    ga.nsplit = static_cast<int>(cdiv(n, kGramRows));
    k_gram_part<<<dim3(ga.nsplit, B), 256, 0, s>>>(ga);
    if (ga.nsplit == 1) return GramOut{g.part, ga.part_bs, 1};
    GramFoldArgs fa;
    fa.part = g.part; fa.part_bs = ga.part_bs; fa.nsplit = ga.nsplit;
    fa.gram = g.gram; fa.gram_bs = sq; fa.l = l;
    k_gram_fold<<<dim3(static_cast<unsigned>(cdiv(static_cast<int64_t>(l) * l, 256)), B), 256, 0, s>>>(fa);
    ++n_fold;
    return GramOut{g.gram, sq, 1};
  };
  if (p.exact) {
    // exact eigenpairs of Gamma = Psi_a Psi_a^T (exact.cu): Q directly, or
    // Q = Psi_a P from the panel P it leaves in y0; then B^T = Psi_a^T Q
    bool project = false;
    if ((e = exact_eigs(g, p, l, mat_ids, count, p.diag, flags, s, prof, &project))) return e;
    if (project && (e = contract(ta, g.y0, g.q))) return e;
    if ((e = contract(tb, g.q, g.bt))) return e;
    prof->begin(kProfEig, s);   // Q K below
  } else {
    // Y0 = Psi_a Omega; p times Y <- Psi_a (Psi_a^T Y)
    if ((e = contract(ta, g.omega, g.y0))) return e;
    float* ycur = g.y0;
    for (int it = 0; it < p.power_iters; ++it) {
      if ((e = contract(tb, ycur, g.zt))) return e;
      if ((e = contract(ta, g.zt, g.y))) return e;
      ycur = g.y;
    }
    // Q = qr(Y): three CholeskyQR passes (the first shifts when its Gram matrix
    // is numerically singular, the others drop numerically dependent
    // columns): y -> q -> zt -> q
    prof->begin(kProfQR, s);
    {
      const float* src = ycur;
      // the first pass's Gram partials by k_gram_part (128-row chunks); the
      // next passes' from the previous solve (256-row chunks); each factor
      // folds its partials itself
      GramArgs ga;
      ga.y = src; ga.y_bs = vbs; ga.part = g.part;
      ga.part_bs = static_cast<int64_t>(g.max_part) * sq;
      ga.n = m_a; ga.l = l;
      ga.nsplit = static_cast<int>(cdiv(m_a, kGramRows));
      k_gram_part<<<dim3(ga.nsplit, B), 256, 0, s>>>(ga);
      NP_CHECK();
      int nsplit = ga.nsplit;
      for (int pass = 0; pass < 3; ++pass) {
        float* dst = (pass == 1) ? g.zt : g.q;
        CholQRArgs cq;
        cq.part = g.part; cq.part_bs = ga.part_bs; cq.nsplit = nsplit;
        cq.gram_out = pass < 2 ? g.part : nullptr;
        cq.gram_bs = ga.part_bs;
        cq.y = src; cq.q = dst; cq.v_bs = vbs;
        cq.n = m_a; cq.l = l; cq.flags = flags;
        cq.vec = (l % 4 == 0) && (vbs % 4 == 0) && (reinterpret_cast<uintptr_t>(src) % 16 == 0) &&
                 (reinterpret_cast<uintptr_t>(dst) % 16 == 0);
        cq.drop = (pass > 0);
        if ((e = launch_cholqr(cq, g.rfac, B, lp, s))) return e;
        src = dst;
        nsplit = static_cast<int>(cdiv(m_a, 256));
      }
    }
    prof->end(kProfQR, s, 7);
    n_fold = 0;
    // B^T = Psi_a^T Q  [n_a x l];  Gamma_Q = B B^T
    if ((e = contract(tb, g.q, g.bt))) return e;
    prof->begin(kProfEig, s);
    {
      const GramOut go = gram(g.bt, n_a);
      NP_CHECK();
      EigArgs ea;
      ea.part = go.p; ea.part_bs = go.bs; ea.nsplit = go.n;
      ea.ritz = g.ritz; ea.ritz_bs = g.lmax;
      ea.z = g.zvec; ea.z_bs = sq;
      ea.kmat = g.kmat; ea.k_bs = sq;
      ea.stats = g.stats; ea.stats_bs = 8;
      ea.count = count; ea.mat_id = mat_ids;
      ea.l = l; ea.rank = p.rank; ea.k_orient = p.k;
      ea.m_a = m_a; ea.n_a = n_a;
      ea.max_sweeps = p.max_sweeps;
      ea.flags = flags;
      const int jthreads = static_cast<int>(jacobi_threads(l));
      const int nj = (l + 1) & ~1;
      const size_t jsmem = 3 * static_cast<size_t>(nj) * (nj + 1) * sizeof(float);
      k_jacobi<<<B, jthreads, jsmem, s>>>(ea);
      NP_CHECK();
    }
  }
  // K is symmetric (its entries are sums of products taken in the same order
  // for (r, s) and (s, r)), so T_a = Psi_a + (Q K) B = Psi_a + Q (B^T K)^T: the
  // l x l product is applied to the shorter of the two panels, Q [m_a x l] or
  // B^T [n_a x l], into g.qk
  const bool k_on_b = n_a < m_a;
  {
    RowMulArgs rm;
    rm.y = k_on_b ? g.bt : g.q; rm.y_bs = vbs; rm.s = g.kmat; rm.s_bs = sq;
    rm.out = g.qk; rm.out_bs = vbs; rm.n = k_on_b ? n_a : m_a; rm.l = l;
    k_rowmul<<<dim3(static_cast<unsigned>(cdiv(rm.n * ((l + 7) / 8), 256)), B), 256, 0, s>>>(rm);
    NP_CHECK();
  }
  prof->end(kProfEig, s, (p.exact ? 1 : 3) + n_fold);
  // T_s = Psi + Lm R^T with (Lm, R) = (QK, B^T) row-active or (B^T, QK)
  // column-active; (Q, B^T K) and (B^T K, Q) when K went on B^T.  In launches
  // of at most kMaxBatch matrices (W pointers travel as kernel arguments)
  const float* u_a = k_on_b ? g.q : g.qk;    // the m_a-row factor
  const float* u_b = k_on_b ? g.qk : g.bt;   // the n_a-row factor
  prof->begin(kProfApplyL, s);
  int n_apply = 0;
  const bool vec = (g.cols % 4 == 0) && (g.ld % 4 == 0);
  for (int c0 = 0; c0 < B; c0 += kMaxBatch) {
    const int nb = std::min(kMaxBatch, B - c0);
    ++n_apply;
    LApplyArgs la;
    std::memset(static_cast<void*>(&la), 0, sizeof(la));   // unused W / G slots are null, never stale
    la.psi = g.psi_bf16 ? static_cast<const void*>(reinterpret_cast<const bf16*>(g.psi) + c0 * psi_bs)
                        : static_cast<const void*>(g.psi + c0 * psi_bs);
    la.psi_bs = psi_bs; la.psi_ld = g.ld; la.psi_bf16 = g.psi_bf16 ? 1 : 0;
    la.lm = (rows_active ? u_a : u_b) + c0 * vbs; la.lm_bs = vbs;
    la.rm = (rows_active ? u_b : u_a) + c0 * vbs; la.rm_bs = vbs;
    la.stats = g.stats + c0 * 8; la.stats_bs = 8;
    for (int i = 0; i < nb; ++i) la.W[i] = W[c0 + i];
    la.rows = g.rows; la.cols = g.cols; la.l = l;
    la.lr = p.lr; la.wd = p.wd; la.target = p.target;
    la.vec_panels = (l % 4 == 0) && (vbs % 4 == 0) &&
                    (reinterpret_cast<uintptr_t>(la.lm) % 16 == 0) && (reinterpret_cast<uintptr_t>(la.rm) % 16 == 0);
    const bool diag = p.diag && p.G;
    la.g_dtype = p.g_dtype;
    for (int i = 0; i < nb; ++i) {
      la.G[i] = diag ? p.G[c0 + i] : nullptr;
      la.diag[i] = diag ? p.diag + 8 * static_cast<int64_t>(p.mat_ids_host[c0 + i]) : nullptr;
    }
    if (!diag && l % 4 == 0 && l <= 64 && la.vec_panels) {
      // tensor-core apply: one persistent CTA per SM over the launch's units
      const int natoms = (l + 31) / 32;
      // the two-atom size for every l: one CTA per SM, so the 512 TMEM
      // columns of a CTA never wait for another's
      const size_t smem = atc_smem(2);
      static bool attr_set[4] = {false, false, false, false};
      const int kind = 2 * (g.w_dtype != 0) + (g.psi_bf16 ? 1 : 0);
      auto go = [&](auto* tw, auto* tp) -> cudaError_t {
        using TWT = std::remove_pointer_t<decltype(tw)>;
        using TPT = std::remove_pointer_t<decltype(tp)>;
        if (!attr_set[kind]) {
          const cudaError_t ea = cudaFuncSetAttribute(k_apply_tc<TWT, TPT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                      static_cast<int>(smem));
          if (ea != cudaSuccess) return ea;
          attr_set[kind] = true;
        }
        const int64_t units = cdiv(g.rows, kAtcRows) * cdiv(g.cols, kAtcCols) * nb;
        const unsigned ctas = static_cast<unsigned>(std::min<int64_t>(units, device_sm_count()));
        k_apply_tc<TWT, TPT><<<ctas, kAtcThreads, smem, s>>>(la, nb, natoms, flags);
        return cudaGetLastError();
      };
      switch (kind) {
        case 0: e = go((float*)nullptr, (float*)nullptr); break;
        case 1: e = go((float*)nullptr, (bf16*)nullptr); break;
        case 2: e = go((bf16*)nullptr, (float*)nullptr); break;
        default: e = go((bf16*)nullptr, (bf16*)nullptr); break;
      }
      if (e != cudaSuccess) return e;
      NP_CHECK();
      continue;
    }
    const dim3 grid(static_cast<unsigned>(cdiv(g.cols, 64)), static_cast<unsigned>(cdiv(g.rows, 64)), nb);
#define NP_APPLY_L(TWT, V) \
    (diag ? k_apply_l<TWT, V, true><<<grid, 256, 0, s>>>(la) : k_apply_l<TWT, V, false><<<grid, 256, 0, s>>>(la))
    if (g.w_dtype == 0) {
      if (vec) NP_APPLY_L(float, true);
      else NP_APPLY_L(float, false);
    } else {
      if (vec) NP_APPLY_L(bf16, true);
      else NP_APPLY_L(bf16, false);
    }
#undef NP_APPLY_L
    NP_CHECK();
  }
  prof->end(kProfApplyL, s, n_apply);
#undef NP_CHECK
  return cudaSuccess;
}

}  // namespace normpre

// ---------------------------------------------------------------------------
// Stand-alone sketch matrix (normpre_sketch_omega): the kernel the step uses,
// for one matrix, with its Philox words and uniforms written out as well.
// ---------------------------------------------------------------------------
extern "C" int normpre_sketch_omega(uint64_t seed, int matrix_id, int64_t t, int64_t n_a, int l, float* omega,
                                    uint32_t* words, float* uniforms, void* stream) {
  using namespace normpre;
  if (!omega) { set_thread_error("null omega pointer"); return NORMPRE_ERR_ARG; }
  if (matrix_id < 0) { set_thread_error("matrix_id must be >= 0"); return NORMPRE_ERR_ARG; }
  if (n_a < 1 || l < 1 || n_a > (int64_t(1) << 24) || l > 4096 || n_a * l > (int64_t(1) << 32)) {
    set_thread_error("n_a and l must be >= 1 with n_a * l <= 2^32 (the 32-bit block counter)");
    return NORMPRE_ERR_SHAPE;
  }
  auto al4 = [](const void* q) { return (reinterpret_cast<uintptr_t>(q) & 3u) == 0; };
  if (!al4(omega) || (words && !al4(words)) || (uniforms && !al4(uniforms))) {
    set_thread_error("outputs must be 4-byte aligned");
    return NORMPRE_ERR_ALIGN;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  OmegaArgs o;
  o.omega = omega; o.bstride = n_a * l; o.n_a = n_a; o.l = l;
  o.key0 = static_cast<uint32_t>(seed); o.key1 = static_cast<uint32_t>(seed >> 32);
  o.t_lo = static_cast<uint32_t>(static_cast<uint64_t>(t)); o.t_hi = static_cast<uint32_t>(static_cast<uint64_t>(t) >> 32);
  o.mat_id = nullptr;
  o.mat_id0 = matrix_id;
  o.words = words;
  o.uniforms = uniforms;
  const int64_t blocks = cdiv(n_a * l, 4);
  k_omega<<<dim3(static_cast<unsigned>(cdiv(blocks, 256)), 1), 256, 0, s>>>(o);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) { set_thread_error(std::string("launch: ") + cudaGetErrorString(e)); return NORMPRE_ERR_CUDA; }
  return NORMPRE_OK;
}
