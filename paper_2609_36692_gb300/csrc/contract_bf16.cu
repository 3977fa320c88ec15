// Sketch contractions with a bf16 Psi (NormPre-L in NORMPRE_PREC_BF16, the
// pure-bf16 setting of the paper's Qwen3 runs, App. A): out = op(Psi) V with
// op(Psi) = Psi (contraction over the stored columns, Y = Psi_a Omega for the
// row-active side) or Psi^T (over the stored rows), V an fp32 [K x l] panel.
//
// Psi is exact in bf16, so one tcgen05 kind::f16 product per K step keeps
// the whole contraction at fp32-accumulated bf16 x (V hi + V lo) precision:
// V is split once per contraction into hi = bf16(V) and lo = bf16(V - hi)
// (together ~2^-16 of V), stacked as the N = 2 np rows of the B operand
// (np = l rounded up to 16), and the drain adds accumulator columns n and
// np + n.  Against the fp32 three-product path this halves the HBM bytes of
// Psi, removes the operand split from the kernel (the Psi tiles go from TMA
// straight to the MMA) and issues a quarter of the MMA instructions.
//
// The TMEM accumulator is not drained mid-unit: its fp32 sums lose at most
// an ulp per addition (~K / 16 ulps over a unit), far below Psi's own bf16
// rounding.
#include <cstring>

#include "common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace normpre {

// ---------------------------------------------------------------------------
// V [K x l] fp32 (row stride l) -> vb [2 np][kpad] bf16: row n < np holds
// hi(V[:, n]), row np + n holds lo(V[:, n]); columns n >= l and K rows >= K
// are zero.  One CTA per 256 K rows of a matrix, in four 64-row blocks each
// staged in shared memory so that both the read and the transposed write are
// coalesced; a thread writes eight K entries of one row as one 16-byte store.
// ---------------------------------------------------------------------------
struct VSplitArgs {
  const float* v; int64_t v_bs;
  int64_t K;
  int l, np;
  bf16* vb; int64_t vb_bs, kpad;
};
static_assert(sizeof(VSplitArgs) + 64 <= 4096, "kernel arguments beyond 4 KB");
constexpr int kVsRows = 256;
__global__ void __launch_bounds__(256) k_vsplit_bf(const __grid_constant__ VSplitArgs a) {
  __shared__ float tile[64][64 + 1];
  const int b = blockIdx.y, tid = threadIdx.x;
  const int l = a.l;   // <= 64
  for (int blk = 0; blk < kVsRows / 64; ++blk) {
    const int64_t k0 = static_cast<int64_t>(blockIdx.x) * kVsRows + 64 * blk;
    if (k0 >= a.kpad) break;
    const float* v = a.v + b * a.v_bs + k0 * l;
    const int64_t left = a.K - k0;
    const int nvalid = left <= 0 ? 0 : static_cast<int>((left < 64 ? left : 64) * l);   // contiguous floats
    if (blk) __syncthreads();          // the previous block's tile is read
    if ((l & 3) == 0 && (reinterpret_cast<uintptr_t>(v) & 15) == 0) {
      for (int i4 = tid; i4 < 16 * l; i4 += 256) {          // 64 l / 4 float4s
        const int i = 4 * i4;
        const float4 x = i < nvalid ? __ldg(reinterpret_cast<const float4*>(v) + i4) : make_float4(0.f, 0.f, 0.f, 0.f);
        const int k = i / l, n = i - k * l;                   // l % 4 == 0: the 4 values share row k
        tile[k][n] = x.x; tile[k][n + 1] = x.y; tile[k][n + 2] = x.z; tile[k][n + 3] = x.w;
      }
    } else {
      for (int i = tid; i < 64 * l; i += 256) {
        const int k = i / l, n = i - k * l;
        tile[k][n] = i < nvalid ? v[i] : 0.f;
      }
    }
    __syncthreads();
    // thread: row n = item / 8, K entries 8 (item % 8) .. + 7 of the block
    bf16* out = a.vb + b * a.vb_bs + k0;
    for (int item = tid; item < a.np * 8; item += 256) {
      const int n = item >> 3, kk = 8 * (item & 7);
      uint32_t hw[4], lw[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float x0 = n < l ? tile[kk + 2 * e][n] : 0.f, x1 = n < l ? tile[kk + 2 * e + 1][n] : 0.f;
        const bf16 h0 = __float2bfloat16_rn(x0), h1 = __float2bfloat16_rn(x1);
        const bf16 g0 = __float2bfloat16_rn(x0 - __bfloat162float(h0)), g1 = __float2bfloat16_rn(x1 - __bfloat162float(h1));
        hw[e] = static_cast<uint32_t>(__bfloat16_as_ushort(h0)) | (static_cast<uint32_t>(__bfloat16_as_ushort(h1)) << 16);
        lw[e] = static_cast<uint32_t>(__bfloat16_as_ushort(g0)) | (static_cast<uint32_t>(__bfloat16_as_ushort(g1)) << 16);
      }
      *reinterpret_cast<uint4*>(out + static_cast<int64_t>(n) * a.kpad + kk) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
      *reinterpret_cast<uint4*>(out + static_cast<int64_t>(a.np + n) * a.kpad + kk) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
    }
  }
}

// ---------------------------------------------------------------------------
// The contraction.  Persistent, one CTA per SM over the units (matrix, K
// split, 128-row tile of the output), matrix-major so that consecutive units
// share V in L2.  Warp 0 issues the TMA copies of each 64-deep K block (the
// Psi tile as two 64 x 64 boxes, K-major for Psi and MN-major for Psi^T; the
// split V as one box of 2 np rows) into a 6-stage ring; warp 1 issues four
// M = 128, N = 2 np, K = 16 MMAs per block into one of two TMEM accumulators
// (128 columns each) and frees the stage; warps 2-5, one per TMEM lane
// quarter, drain a finished accumulator into the unit's rows while the next
// unit accumulates in the other.
// ---------------------------------------------------------------------------
constexpr int kCbStages = 6;
constexpr int kCbA = 128 * 128;                 // 128 rows x 64 K bf16
constexpr int kCbB = 128 * 128;                 // up to 128 rows (V hi | V lo) x 64 K bf16
constexpr int kCbStage = kCbA + kCbB;
constexpr int kCbDrainWarps = 4;
constexpr int kCbThreads = 64 + 32 * kCbDrainWarps;
constexpr size_t kCbSmem = 1024 + static_cast<size_t>(kCbStages) * kCbStage + 256;
constexpr uint32_t kCbTmemCols = 256;

struct ContractBfArgs {
  CUtensorMap psi_map;    // bf16 {cols, rows, batch}, box 64 x 64, 128-byte swizzle
  CUtensorMap v_map;      // bf16 {kpad, 2 np, batch}, box 64 x 2 np
  float* out; int64_t out_bs;
  int64_t P, K;
  int l, np;
  int64_t kchunk;         // K range of one split (multiple of 64)
  int ksplit, batch;
  int* flags;
  int stall_first_copy;   // tests: CTA 0 does not issue its first copy (its waits then give up)
};
static_assert(sizeof(ContractBfArgs) + 64 <= 4096, "kernel arguments beyond 4 KB");

template <bool TRANS>
__global__ void __launch_bounds__(kCbThreads, 1) k_contract_bf(const __grid_constant__ ContractBfArgs a) {
  extern __shared__ uint8_t cb_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(cb_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kCbStages * kCbStage);   // [kCbStages] copies landed
  uint64_t* empty = full + kCbStages;                                          // [kCbStages] MMAs done
  uint64_t* tfull = empty + kCbStages;                                         // [2] unit accumulated
  uint64_t* tempty = tfull + 2;                                                // [2] accumulator drained
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint32_t* issued = reinterpret_cast<uint32_t*>(tmem_slot + 2);              // [kCbStages] last parity + 1

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tiles = static_cast<int>((a.P + 127) / 128);
  const int units = tiles * a.ksplit * a.batch;
  auto unit_of = [&](int u, int& b, int& z, int64_t& p0, int64_t& kbeg, int& nk) {
    p0 = static_cast<int64_t>(u % tiles) * 128;
    z = (u / tiles) % a.ksplit;
    b = u / (tiles * a.ksplit);
    kbeg = static_cast<int64_t>(z) * a.kchunk;
    const int64_t kend = min(a.K, kbeg + a.kchunk);
    nk = kend > kbeg ? static_cast<int>((kend - kbeg + 63) / 64) : 0;
  };
  if (threadIdx.x == 0) {
    for (int i = 0; i < kCbStages; ++i) {
      tc::mbar_init(&full[i], 1);
      tc::mbar_init(&empty[i], 1);
      issued[i] = 0;
    }
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&tfull[i], 1);
      tc::mbar_init(&tempty[i], kCbDrainWarps);
    }
    *abort_flag = 0;
    tc::fence_barrier_init();
    tc::prefetch_map(&a.psi_map);
    tc::prefetch_map(&a.v_map);
  }
  if (warp == 1) {
    tc::tmem_alloc(tmem_slot, kCbTmemCols);
    tc::tmem_relinquish();
    tc::fence_before();
  }
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t vbytes = static_cast<uint32_t>(2 * a.np * 128);

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    bool ok = true;
    uint32_t it = 0;
    for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
      int b, z, nk;
      int64_t p0, kbeg;
      unit_of(u, b, z, p0, kbeg, nk);
      for (int kb = 0; kb < nk && ok; ++kb, ++it) {
        const int i = it % kCbStages;
        const uint32_t ph = (it / kCbStages) & 1;
        ok = __all_sync(0xffffffffu, tc::mbar_wait(&empty[i], ph ^ 1u, abort_flag));
        if (!ok) break;
        if (lane == 0 && !(a.stall_first_copy && blockIdx.x == 0 && it == 0)) {
          tc::mbar_expect_tx(&full[i], static_cast<uint32_t>(kCbA) + vbytes);
          issued[i] = ph + 1;
          uint8_t* st = smem + i * kCbStage;
          const int k0 = static_cast<int>(kbeg) + 64 * kb, pr = static_cast<int>(p0);
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            if (!TRANS) tc::tma_load_3d(st + j * 8192, &a.psi_map, &full[i], k0, pr + 64 * j, b);
            else        tc::tma_load_3d(st + j * 8192, &a.psi_map, &full[i], pr + 64 * j, k0, b);
          }
          tc::tma_load_3d(st + kCbA, &a.v_map, &full[i], k0, 0, b);
        }
        __syncwarp();
      }
    }
    if (!ok && lane == 0) { *abort_flag = 1; raise_flag(a.flags, kFlagTimeout); }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    const uint32_t idesc = tc::idesc_bf16(128, 2 * a.np, TRANS ? 1 : 0, 0);
    // descriptor steps per 16-deep K slice: K-major +32 B, MN-major +2048 B
    // (8-row K groups of 1024 B; the two 64-wide MN halves 8 KB apart)
    const uint32_t a_step = TRANS ? 2048u : 32u, a_lbo = TRANS ? 8192u : 16u;
    bool ok = true;
    uint32_t it = 0, ga = 0;   // stage counter; accumulator counter over the units with K work
    for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
      int b, z, nk;
      int64_t p0, kbeg;
      unit_of(u, b, z, p0, kbeg, nk);
      if (nk == 0) continue;
      const int acc = ga & 1;
      ok = __all_sync(0xffffffffu, tc::mbar_wait(&tempty[acc], ((ga >> 1) & 1) ^ 1u, abort_flag));
      if (!ok) break;
      tc::fence_after();
      const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(128 * acc);
      for (int kb = 0; kb < nk && ok; ++kb, ++it) {
        const int i = it % kCbStages;
        const uint32_t ph = (it / kCbStages) & 1;
        ok = __all_sync(0xffffffffu, tc::mbar_wait(&full[i], ph, abort_flag));
        if (!ok) break;
        tc::fence_after();
        if (lane == 0) {
          const uint32_t sa = tc::su32(smem + i * kCbStage), sb = sa + kCbA;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            const uint64_t ad = tc::sdesc(sa + kk * a_step, a_lbo, 1024);
            const uint64_t bd = tc::sdesc(sb + kk * 32, 16, 1024);
            tc::mma_bf16(d_tmem, ad, bd, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
          }
          tc::mma_commit(&empty[i]);
          if (kb == nk - 1) tc::mma_commit(&tfull[acc]);
        }
        __syncwarp();
      }
      ++ga;
    }
    if (!ok && lane == 0) { *abort_flag = 1; raise_flag(a.flags, kFlagTimeout); }
  } else {
    // ---------------- drains (warps 2..5): out row = 32 q + lane of the unit ----------------
    const int q = warp & 3;
    bool ok = true;
    uint32_t ga = 0;
    for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
      int b, z, nk;
      int64_t p0, kbeg;
      unit_of(u, b, z, p0, kbeg, nk);
      const int64_t row = p0 + 32 * q + lane;
      float* out = a.out + b * a.out_bs + static_cast<int64_t>(z) * a.P * a.l + row * a.l;
      if (nk == 0) {
        if (row < a.P)
          for (int j = 0; j < a.l; ++j) out[j] = 0.f;
        continue;
      }
      const int acc = ga & 1;
      ok = __all_sync(0xffffffffu, tc::mbar_wait(&tfull[acc], (ga >> 1) & 1, abort_flag));
      if (!ok) break;
      tc::fence_after();
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        if (16 * h < a.np) {
          uint32_t r[16], v[16];
          const uint32_t col = tmem_base + (static_cast<uint32_t>(32 * q) << 16) + static_cast<uint32_t>(128 * acc + 16 * h);
          tc::tmem_ld16(col, r);
          tc::tmem_ld16(col + static_cast<uint32_t>(a.np), v);
          tc::tmem_ld_wait();
          if (row < a.P) {
#pragma unroll
            for (int j = 0; j < 16; ++j)
              if (16 * h + j < a.l) out[16 * h + j] = __uint_as_float(r[j]) + __uint_as_float(v[j]);
          }
        }
      }
      tc::fence_before();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&tempty[acc]);
      ++ga;
    }
    if (!ok && lane == 0) { *abort_flag = 1; raise_flag(a.flags, kFlagTimeout); }
  }
  __syncthreads();
  if (threadIdx.x == 0 && *abort_flag) {
    // let every TMA copy still in flight land before the CTA exits
    volatile int never = 0;
    for (int i = 0; i < kCbStages; ++i)
      if (issued[i]) tc::mbar_wait(&full[i], issued[i] - 1, &never);
  }
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::fence_after();
    tc::tmem_dealloc(tmem_base, kCbTmemCols);
  }
}

bool contract_bf16_map(CUtensorMap* map, const void* psi, int64_t rows, int64_t cols, int64_t ld, int batch,
                       int box_rows) {
  const uint64_t dims[3] = {static_cast<uint64_t>(cols), static_cast<uint64_t>(rows), static_cast<uint64_t>(batch)};
  const uint64_t strides[2] = {static_cast<uint64_t>(ld) * 2, static_cast<uint64_t>(rows * ld) * 2};
  const uint32_t box[3] = {64, static_cast<uint32_t>(box_rows), 1};
  return (ld % 8 == 0) &&
         driver_encode_tiled(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(psi), dims, strides, box, nullptr);
}

cudaError_t launch_contract_bf16(const ContractBf16Launch& c, cudaStream_t s) {
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_contract_bf<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(kCbSmem));
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(k_contract_bf<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(kCbSmem));
    if (e != cudaSuccess) return e;
    attr = true;
  }
  if (c.l < 1 || c.l > 64) return cudaErrorInvalidValue;
  const int np = static_cast<int>(round_up(c.l, 16));
  const int64_t kpad = round_up(c.K, 64);
  if (2 * np * kpad > c.vb_bs) return cudaErrorInvalidValue;
  // V hi / lo, transposed to K-major bf16 rows
  VSplitArgs vs;
  vs.v = c.v; vs.v_bs = c.v_bs; vs.K = c.K; vs.l = c.l; vs.np = np;
  vs.vb = static_cast<bf16*>(c.vb); vs.vb_bs = c.vb_bs; vs.kpad = kpad;
  k_vsplit_bf<<<dim3(static_cast<unsigned>(cdiv(kpad, kVsRows)), static_cast<unsigned>(c.batch)), 256, 0, s>>>(vs);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  ContractBfArgs a;
  std::memset(static_cast<void*>(&a), 0, sizeof(a));
  a.psi_map = *c.psi_map;
  const uint64_t vdims[3] = {static_cast<uint64_t>(kpad), static_cast<uint64_t>(2 * np), static_cast<uint64_t>(c.batch)};
  const uint64_t vstr[2] = {static_cast<uint64_t>(kpad) * 2, static_cast<uint64_t>(c.vb_bs) * 2};
  const uint32_t vbox[3] = {64, static_cast<uint32_t>(2 * np), 1};
  if (!driver_encode_tiled(&a.v_map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, c.vb, vdims, vstr, vbox, nullptr))
    return cudaErrorInvalidValue;
  a.out = c.out; a.out_bs = c.out_bs;
  a.P = c.P; a.K = c.K; a.l = c.l; a.np = np;
  a.kchunk = c.kchunk; a.ksplit = c.ksplit; a.batch = c.batch;
  a.flags = c.flags;
  a.stall_first_copy = c.stall_first_copy;
  const int64_t units = cdiv(c.P, 128) * c.ksplit * c.batch;
  const unsigned grid = static_cast<unsigned>(std::min<int64_t>(units, device_sm_count()));
  if (c.trans) k_contract_bf<true><<<grid, kCbThreads, kCbSmem, s>>>(a);
  else k_contract_bf<false><<<grid, kCbThreads, kCbSmem, s>>>(a);
  return cudaGetLastError();
}

}  // namespace normpre
