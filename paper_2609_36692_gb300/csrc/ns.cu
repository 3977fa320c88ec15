// Newton-Schulz preconditioner of NormPre-G (Sec. 3.2 and App. B of the paper;
// the iteration is Muon's: X <- a X + (b A + c A^2) X with A = X X^T, after
// scaling X to unit Frobenius norm, and with the input transposed when it has
// more rows than columns so that the Gram matrix is s x s, App. C).
//
// GB300 design:
//   * Every matrix stays in its stored (row-major) layout.  A "wide" matrix
//     (rows <= cols) has Gram X X^T; a "tall" one X^T X.  Instead of
//     transposing, the GEMMs read operands either K-major or MN-major straight
//     from the layout they are in (the tcgen05 instruction descriptor's
//     transpose bits and the matching shared-memory descriptors).
//   * Each of the three products of an iteration is one persistent launch over
//     all shape groups and all matrices of a group (grouped GEMM): one CTA per
//     SM walks a static list of 128 x BN output tiles.
//   * bf16 path: TMA (cp.async.bulk.tensor, 128-byte swizzle) feeds a 4-stage
//     shared-memory ring; one thread issues tcgen05.mma (kind::f16, bf16 in,
//     fp32 accumulate) into a double-buffered TMEM accumulator; four epilogue
//     warps read TMEM with tcgen05.ld and fuse the polynomial combine, the
//     1/||Psi||_F prescale of the first iteration and the ||T||_F^2 partial
//     sums of the last one.
//   * The iteration is evaluated as X <- C X with C = a I + b A + c A^2 formed
//     (in fp32, rounded once) by the epilogue of the A A product.  For singular
//     values near the quintic's fixed band a X and B X nearly cancel, so adding
//     them after rounding B to bf16 would amplify B's rounding error; folding
//     a I into C keeps every stored operand's relative error at one rounding
//     and spares the update epilogue a read of X.
//   * fp32 path (parity mode): a plain SIMT tiled GEMM with the same epilogues.
//   * Zero padding (dims rounded up to the tile) is preserved by every product,
//     so tiles never need bounds checks.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstring>

#include "common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace normpre {

// ---------------------------------------------------------------------------
// Driver entry point for tensor-map encoding (no link-time libcuda dependency).
// ---------------------------------------------------------------------------
bool driver_encode_tiled(CUtensorMap* map, CUtensorMapDataType dt, uint32_t rank, void* addr,
                         const uint64_t* dims, const uint64_t* strides_bytes, const uint32_t* box,
                         std::string* err) {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                                     cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !p) {
      if (err) *err = "cuTensorMapEncodeTiled entry point unavailable";
      return false;
    }
    fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  cuuint64_t d[5], st[4];
  cuuint32_t bx[5], es[5];
  for (uint32_t i = 0; i < rank; ++i) { d[i] = dims[i]; bx[i] = box[i]; es[i] = 1; }
  for (uint32_t i = 0; i + 1 < rank; ++i) st[i] = strides_bytes[i];
  CUresult r = fn(map, dt, rank, addr, d, st, bx, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (err) *err = "cuTensorMapEncodeTiled failed with CUresult " + std::to_string((int)r);
    return false;
  }
  return true;
}

int device_sm_count() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}


// ---------------------------------------------------------------------------
// Grouped GEMM description shared by the tensor-core and SIMT kernels.
//   C[b](i, j) = sum_k A_b(i, k) B_b(j, k)
//   A_b(i, k) = a_mn ? Abuf_b[k][i] : Abuf_b[i][k]     (likewise B)
//   out = s * (ca * aux(i, j) + cb * C(i, j) + (i == j ? diag : 0)),
//   s = inscale[b]^scale_pow
// ---------------------------------------------------------------------------
struct GemmGroup {
  CUtensorMap mapA;            // tensor-core path only (3-D, box 64 x 64 x 1)
  CUtensorMap mapB;
  const void* Abuf;            // SIMT path: operand bases
  const void* Bbuf;
  int64_t a_ld, a_bs, b_ld, b_bs;
  int a_mn, b_mn;
  int M, N, K, BN;
  int batch, tiles_m, tiles_n, tile_begin;
  int b_base;                  // index in the group of this launch's first matrix
  int sym;                     // symmetric output: only tiles reaching the diagonal, mirrored
  int per;                     // tiles per matrix
  float ca, cb, diag;
  int scale_pow;
  void* out;
  int64_t out_ld, out_bs;
  const void* aux;
  int64_t aux_ld, aux_bs;
  const float* inscale;
  float* sq_part;              // [batch][tiles_m * tiles_n * parts_per_tile] or null
};
struct GemmArgs {
  GemmGroup g[kMaxGroups];
  int n_groups;
  int total_tiles;
  int* flags;
};
static_assert(sizeof(GemmArgs) + 64 <= 4096, "kernel arguments beyond 4 KB");

// Tiles of one matrix: the whole tiles_m x tiles_n grid, or for a symmetric
// product only the tiles that reach the diagonal or lie above it
// (tm <= (BN / 128)(tn + 1) - 1), enumerated column by column.
__host__ __device__ inline int tiles_per_matrix(int tiles_m, int tiles_n, int bn, int sym) {
  if (!sym) return tiles_m * tiles_n;
  const int rr = bn / 128;
  int n = 0;
  for (int tn = 0; tn < tiles_n; ++tn) n += (rr * (tn + 1) < tiles_m) ? rr * (tn + 1) : tiles_m;
  return n;
}

// Work unit t -> (group, matrix b, row tile tm, column tile tn).  With
// pairs = 1 a unit is two vertically adjacent tiles (2p, tn) and (2p + 1, tn)
// that share their B operand, one per CTA of a cluster (`sub` = 0 or 1); every
// group then has an even number of row tiles.
__device__ __forceinline__ int decode_tile(const GemmArgs& a, int t, int& b, int& tm, int& tn, int pairs = 0,
                                           int sub = 0) {
  int gi = 0;
  for (; gi < a.n_groups - 1; ++gi) {
    const GemmGroup& g = a.g[gi];
    if (t < ((g.tile_begin + g.batch * g.per) >> pairs)) break;
  }
  const GemmGroup& g = a.g[gi];
  const int per = g.per >> pairs;
  const int l = t - (g.tile_begin >> pairs);
  b = l / per;
  int r = l - b * per;
  b += g.b_base;
  if (!g.sym) {
    const int tmu = r / g.tiles_n;
    tn = r - tmu * g.tiles_n;
    tm = (tmu << pairs) + sub;
  } else {
    const int rr = g.BN / 128;
    int c = 0;
    for (;; ++c) {
      const int cnt = ((rr * (c + 1) < g.tiles_m) ? rr * (c + 1) : g.tiles_m) >> pairs;
      if (r < cnt) break;
      r -= cnt;
    }
    tm = (r << pairs) + sub;
    tn = c;
  }
  return gi;
}

// ---------------------------------------------------------------------------
// tcgen05 grouped GEMM
// ---------------------------------------------------------------------------
constexpr int kBM = 128, kBK = 64, kStages = 4;
constexpr int kStageA = kBM * kBK * 2;   // 16 KB
constexpr int kStageB = 256 * kBK * 2;   // 32 KB (BN <= 256)
constexpr int kEpiWarps = 8;             // two per TMEM lane quarter, each with half the columns
constexpr int kTcThreads = 64 + 32 * kEpiWarps;   // warp 0 TMA, warp 1 MMA, then the epilogue
constexpr int kTmemCols = 512;           // two 128 x 256 fp32 accumulators
// Per epilogue warp: two 32 x 32 bf16 staging blocks (the chunk as computed
// and its transpose), 64-byte rows whose 16-byte pieces are XOR-swizzled by
// (row >> 1) & 3 so that both row-per-lane and 8-rows-per-instruction
// accesses are free of bank conflicts.
constexpr size_t kStageBlockBytes = 32 * 32 * 2;
constexpr size_t kEpiBytes = kEpiWarps * 2 * kStageBlockBytes;
constexpr size_t kTcSmem = 1024 + kStages * (kStageA + kStageB) + 256 + kEpiBytes;

// Staging block accessors: row r (0..31), 16-byte piece p (0..3) of a 32 x 32
// bf16 block with 64-byte rows; the piece is stored at p ^ ((r >> 1) & 3).
__device__ __forceinline__ uint32_t stage_off(int r, int p) {
  return static_cast<uint32_t>(r * 64 + ((p ^ ((r >> 1) & 3)) << 4));
}
__device__ __forceinline__ void stage_st(uint8_t* blk, int r, int p, uint4 v) {
  *reinterpret_cast<uint4*>(blk + stage_off(r, p)) = v;
}
__device__ __forceinline__ uint4 stage_ld(const uint8_t* blk, int r, int p) {
  return *reinterpret_cast<const uint4*>(blk + stage_off(r, p));
}
__device__ __forceinline__ void stage_st16(uint8_t* blk, int r, int col, uint16_t v) {
  *reinterpret_cast<uint16_t*>(blk + stage_off(r, col >> 3) + 2 * (col & 7)) = v;
}

// Stores the diagonal 32 x 32 block of a symmetric product: from the chunk
// (stg) the elements on or above the diagonal, from its transpose (tbuf) the
// ones below it, so the block is exactly symmetric.  Lane -> rows crow + 8 i,
// columns 8 cpiece .. + 7.  Out of line: it runs for few chunks.
__device__ __noinline__ void store_diag_block(const uint8_t* stg, const uint8_t* tbuf, bf16* outb, int64_t out_ld,
                                              int64_t r0, int64_t c0, int crow, int cpiece) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int rr = crow + 8 * i;
    const uint4 a = stage_ld(stg, rr, cpiece), t = stage_ld(tbuf, rr, cpiece);
    const uint32_t a4[4] = {a.x, a.y, a.z, a.w}, t4[4] = {t.x, t.y, t.z, t.w};
    uint32_t o4[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int c = 8 * cpiece + 2 * e;   // columns c, c + 1 of row rr
      const uint32_t lo = (c >= rr ? a4[e] : t4[e]) & 0xFFFFu;
      const uint32_t hi = (c + 1 >= rr ? a4[e] : t4[e]) & 0xFFFF0000u;
      o4[e] = lo | hi;
    }
    *reinterpret_cast<uint4*>(outb + (r0 + rr) * out_ld + c0 + 8 * cpiece) = make_uint4(o4[0], o4[1], o4[2], o4[3]);
  }
}

// Keeps a per-tile parameter in a register: the group descriptors live in the
// kernel's parameter space and are indexed at run time, and a plain copy may
// be re-read from there after every asm statement that clobbers memory.
__device__ __forceinline__ int pin(int v) { asm volatile("" : "+r"(v)); return v; }
__device__ __forceinline__ int64_t pin(int64_t v) { asm volatile("" : "+l"(v)); return v; }
__device__ __forceinline__ float pin(float v) { asm volatile("" : "+f"(v)); return v; }
template <typename T>
__device__ __forceinline__ T* pin(T* v) {
  uint64_t u = reinterpret_cast<uint64_t>(v);
  asm volatile("" : "+l"(u));
  return reinterpret_cast<T*>(u);
}

// MC = false: each CTA computes its own 128 x BN tiles.
// MC = true: clusters of two CTAs take units of two vertically adjacent tiles
// with the same B operand; each CTA loads its own A rows and half of B,
// multicasting that half into both CTAs, so a CTA reads 16 + BN/128 * 16 KB
// per 64-deep K block from L2 instead of 16 + BN/64 * 16 KB.  A stage is
// refilled only after the MMAs of both CTAs released it.
template <bool MC>
__global__ void __launch_bounds__(kTcThreads, 1) k_ns_gemm_tc(const __grid_constant__ GemmArgs args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + kStages * kStageA;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + kStages * kStageB);
  uint64_t* empty = full + kStages;
  uint64_t* tfull = empty + kStages;   // [2]
  uint64_t* tempty = tfull + 2;        // [2]
  uint64_t* drain = tempty + 2;        // [1]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint32_t* issued = reinterpret_cast<uint32_t*>(tmem_slot + 2);   // [kStages] last parity + 1
  uint8_t* epi = sB + kStages * kStageB + 256;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int sub = MC ? static_cast<int>(tc::cluster_rank()) : 0;
  const int unit0 = MC ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
  const int nunits = MC ? static_cast<int>(gridDim.x >> 1) : static_cast<int>(gridDim.x);
  const int units = MC ? (args.total_tiles >> 1) : args.total_tiles;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      tc::mbar_init(&full[s], 1);
      tc::mbar_init(&empty[s], MC ? 2 : 1);   // MC: released by the MMAs of both CTAs
      issued[s] = 0;
    }
    for (int a = 0; a < 2; ++a) {
      tc::mbar_init(&tfull[a], 1);
      tc::mbar_init(&tempty[a], kEpiWarps);
    }
    tc::mbar_init(drain, 1);
    *abort_flag = 0;
    tc::fence_barrier_init();
    for (int gi = 0; gi < args.n_groups; ++gi) {
      tc::prefetch_map(&args.g[gi].mapA);
      tc::prefetch_map(&args.g[gi].mapB);
    }
  }
  if (MC) tc::cluster_sync();   // both CTAs' barriers exist before any multicast reaches them
  if (warp == 1) {
    tc::tmem_alloc(tmem_slot, kTmemCols);
    tc::tmem_relinquish();
    tc::fence_before();
  }
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ---------------- TMA producer (the warp waits, lane 0 issues) ----------------
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    for (int t = unit0; t < units && ok; t += nunits) {
      int b, tm, tn;
      const GemmGroup& g = args.g[decode_tile(args, t, b, tm, tn, MC, sub)];
      const int BN = pin(g.BN), a_mn = pin(g.a_mn), b_mn = pin(g.b_mn);
      const CUtensorMap* mapA = pin(&g.mapA);
      const CUtensorMap* mapB = pin(&g.mapB);
      const int m0 = tm * kBM, n0 = tn * BN, nk = pin(g.K) / kBK;
      // 64-row boxes of B this CTA fetches (MC: its half, for both CTAs)
      const int nbox = BN / 64, bbox0 = MC ? sub * (nbox >> 1) : 0, bbox1 = MC ? bbox0 + (nbox >> 1) : nbox;
      const uint32_t bytes = static_cast<uint32_t>((kBM + BN) * kBK * 2);
      for (int kb = 0; kb < nk; ++kb) {
        ok = __all_sync(0xffffffffu, tc::mbar_wait(&empty[stage], phase ^ 1u, abort_flag));
        if (!ok) break;
        if (lane == 0) {
          tc::mbar_expect_tx(&full[stage], bytes);
          issued[stage] = phase + 1;
          const int k0 = kb * kBK;
          uint8_t* dA = sA + stage * kStageA;
          uint8_t* dB = sB + stage * kStageB;
#pragma unroll
          for (int i = 0; i < kBM / 64; ++i) {
            const int c0 = a_mn ? m0 + 64 * i : k0, c1 = a_mn ? k0 : m0 + 64 * i;
            tc::tma_load_3d(dA + i * 8192, mapA, &full[stage], c0, c1, b);
          }
          for (int i = bbox0; i < bbox1; ++i) {
            const int c0 = b_mn ? n0 + 64 * i : k0, c1 = b_mn ? k0 : n0 + 64 * i;
            if (MC) tc::tma_load_3d_mc(dB + i * 8192, mapB, &full[stage], c0, c1, b, 3);
            else    tc::tma_load_3d(dB + i * 8192, mapB, &full[stage], c0, c1, b);
          }
        }
        __syncwarp();
        if (++stage == kStages) { stage = 0; phase ^= 1u; }
      }
    }
    if (!ok && lane == 0) { *abort_flag = 1; raise_flag(args.flags, kFlagTimeout); }
  } else if (warp == 1) {
    // ---------------- MMA issuer (the warp waits, lane 0 issues) ----------------
    int stage = 0, it = 0;
    uint32_t phase = 0;
    bool ok = true;
    for (int t = unit0; t < units && ok; t += nunits, ++it) {
      int b, tm, tn;
      const GemmGroup& g = args.g[decode_tile(args, t, b, tm, tn, MC, sub)];
      const int nk = pin(g.K) / kBK, a_mn = pin(g.a_mn), b_mn = pin(g.b_mn), BN = pin(g.BN);
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      ok = __all_sync(0xffffffffu, tc::mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag));
      if (!ok) break;
      tc::fence_after();
      const uint32_t idesc = tc::idesc_bf16(kBM, BN, a_mn, b_mn);
      // descriptor steps per 16-deep K slice: K-major +32 B, MN-major +2048 B
      const uint32_t a_step = a_mn ? 2048u : 32u, b_step = b_mn ? 2048u : 32u;
      const uint32_t a_lbo = a_mn ? 8192u : 16u, b_lbo = b_mn ? 8192u : 16u;
      const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * 256);
      for (int kb = 0; kb < nk; ++kb) {
        ok = __all_sync(0xffffffffu, tc::mbar_wait(&full[stage], phase, abort_flag));
        if (!ok) break;
        tc::fence_after();
        if (lane == 0) {
          const uint32_t a_addr = tc::su32(sA + stage * kStageA);
          const uint32_t b_addr = tc::su32(sB + stage * kStageB);
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk) {
            const uint64_t ad = tc::sdesc(a_addr + kk * a_step, a_lbo, 1024);
            const uint64_t bd = tc::sdesc(b_addr + kk * b_step, b_lbo, 1024);
            tc::mma_bf16(d_tmem, ad, bd, idesc, (kb | kk) != 0 ? 1u : 0u);
          }
          if (MC) tc::mma_commit_mc(&empty[stage], 3);
          else tc::mma_commit(&empty[stage]);
        }
        __syncwarp();
        if (++stage == kStages) { stage = 0; phase ^= 1u; }
      }
      if (!ok) break;
      if (lane == 0) tc::mma_commit(&tfull[acc]);
      __syncwarp();
    }
    if (!ok && lane == 0) { *abort_flag = 1; raise_flag(args.flags, kFlagTimeout); }
    // every MMA issued by lane 0 has completed once `drain` fires
    if (lane == 0) {
      tc::mma_commit(drain);
      volatile int never = 0;
      tc::mbar_wait(drain, 0, &never);
    }
    __syncwarp();
  } else {
    // ---------------- epilogue: warps 2..5 ----------------
    const int q = warp & 3;                          // TMEM lane quarter this warp may read
    const int ew = warp - 2;                         // epilogue warp 0 .. kEpiWarps - 1
    const int half = ew >> 2;                        // which half of the tile's columns
    uint8_t* stg = epi + ew * 2 * kStageBlockBytes;  // this warp's chunk, as computed
    uint8_t* tbuf = stg + kStageBlockBytes;          // and transposed
    const int crow = lane >> 2, cpiece = lane & 3;   // coalesced access: rows crow + 8 i, piece cpiece
    int it = 0;
    for (int t = unit0; t < units; t += nunits, ++it) {
      int b, tm, tn;
      const GemmGroup& g = args.g[decode_tile(args, t, b, tm, tn, MC, sub)];
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      const int64_t r0 = static_cast<int64_t>(tm) * kBM + q * 32;   // first row of this warp
      const int64_t row = r0 + lane;
      const int BN = pin(g.BN), sym = pin(g.sym);
      const int64_t out_ld = pin(g.out_ld);
      float* const sq_part = pin(g.sq_part);
      const int64_t n0 = static_cast<int64_t>(tn) * BN;
      bf16* outb = pin(static_cast<bf16*>(g.out) + b * g.out_bs);
      // aux rows are read 8 per instruction: lane -> rows r0 + crow + 8 i, columns n0 + 8 cpiece
      const bf16* auxp = g.aux ? static_cast<const bf16*>(g.aux) + b * g.aux_bs + (r0 + crow) * g.aux_ld + n0 + 8 * cpiece
                               : nullptr;
      auxp = pin(auxp);
      // 32-column chunk kinds (rows r0.. and columns n0 + c.. are both 32-aligned):
      // 0 = store as is (and mirror when symmetric: strictly above the diagonal),
      // 1 = the diagonal 32 x 32 block, 2 = strictly below (written by mirrors).
      auto kind = [&](int c) -> int {
        if (!sym) return 0;
        const int64_t j0 = n0 + c;
        return r0 < j0 ? 0 : (r0 == j0 ? 1 : 2);
      };
      // the aux operand does not depend on the accumulator: fetch the first two
      // chunks before waiting for it
      uint4 ax0[4], ax1[4];   // aux of the next two chunks
      const int64_t aux8 = pin(8 * g.aux_ld);
      const int c_lo = half * (BN >> 1), c_hi = c_lo + (BN >> 1);   // this warp's columns
      auto fetch_aux = [&](int c, uint4 (&dst)[4]) {
        if (auxp && c < c_hi && kind(c) != 2)
#pragma unroll
          for (int i = 0; i < 4; ++i) dst[i] = __ldg(reinterpret_cast<const uint4*>(auxp + i * aux8 + c));
      };
      fetch_aux(c_lo, ax0);
      fetch_aux(c_lo + 32, ax1);
      if (!tc::mbar_wait(&tfull[acc], acc_phase, abort_flag)) {
        *abort_flag = 1;
        raise_flag(args.flags, kFlagTimeout);
        break;
      }
      tc::fence_after();
      float s = 1.f;
      if (g.scale_pow) {
        const float v = g.inscale[b];
        s = g.scale_pow == 2 ? v * v : v;
      }
      const float ca = pin(g.ca * s), cb = pin(g.cb * s), dg = pin(g.diag * s);
      const int64_t diag_col = row - n0;   // column of this thread's diagonal element in the tile
      float sq = 0.f;
      const uint32_t tbase = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * 256);
      // one copy of the chunk code (a small loop body stays in the instruction cache)
#pragma unroll 1
      for (int c = c_lo; c < c_hi; c += 32) {
        const int kd = kind(c);
        uint4 w[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) { w[i] = ax0[i]; ax0[i] = ax1[i]; }
        fetch_aux(c + 64, ax1);
        if (kd == 2) continue;
        uint32_t r[32];
        tc::tmem_ld32(tbase + c, r);
        if (auxp) {
          // regroup the aux block from 8-rows-per-instruction to row-per-lane
#pragma unroll
          for (int i = 0; i < 4; ++i) stage_st(stg, crow + 8 * i, cpiece, w[i]);
          __syncwarp();
#pragma unroll
          for (int v = 0; v < 4; ++v) w[v] = stage_ld(stg, lane, v);
        }
        tc::tmem_ld_wait();
        uint32_t pk[16];
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          float x[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) x[e] = cb * __uint_as_float(r[8 * v + e]);
          if (auxp) {
            const uint32_t w4[4] = {w[v].x, w[v].y, w[v].z, w[v].w};
#pragma unroll
            for (int e = 0; e < 8; ++e)
              x[e] = fmaf(ca, (e & 1) ? bf16hi(w4[e >> 1]) : bf16lo(w4[e >> 1]), x[e]);
          }
          if (kd == 1 && dg != 0.f) {
#pragma unroll
            for (int e = 0; e < 8; ++e)
              if (diag_col == c + 8 * v + e) x[e] += dg;
          }
#pragma unroll
          for (int e = 0; e < 4; ++e) pk[4 * v + e] = pack_bf16x2(x[2 * e], x[2 * e + 1]);
        }
        if (sq_part) {
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const float y0 = bf16lo(pk[e]), y1 = bf16hi(pk[e]);
            sq += y0 * y0 + y1 * y1;
          }
        }
        // each lane owns one row of stg: the aux it read there is replaced by
        // its results without crossing lanes
#pragma unroll
        for (int v = 0; v < 4; ++v) stage_st(stg, lane, v, make_uint4(pk[4 * v], pk[4 * v + 1], pk[4 * v + 2], pk[4 * v + 3]));
        if (sym) {
          // transposed copy: element (lane, e) -> (e, lane)
#pragma unroll
          for (int e = 0; e < 32; ++e)
            stage_st16(tbuf, e, lane, static_cast<uint16_t>((e & 1) ? (pk[e >> 1] >> 16) : (pk[e >> 1] & 0xFFFFu)));
        }
        __syncwarp();
        if (kd == 1) {
          store_diag_block(stg, tbuf, outb, out_ld, r0, n0 + c, crow, cpiece);
        } else {
          // rows r0 + crow + 8 i, columns n0 + c + 8 cpiece .. + 7
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int rr = crow + 8 * i;
            *reinterpret_cast<uint4*>(outb + (r0 + rr) * out_ld + n0 + c + 8 * cpiece) = stage_ld(stg, rr, cpiece);
          }
          if (sym) {
            // mirror: row n0 + c + jj of the output receives column jj of the chunk
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const int jj = crow + 8 * i;
              *reinterpret_cast<uint4*>(outb + (n0 + c + jj) * out_ld + r0 + 8 * cpiece) = stage_ld(tbuf, jj, cpiece);
            }
          }
        }
        __syncwarp();   // stg / tbuf are rewritten by the next chunk
      }
      tc::fence_before();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&tempty[acc]);
      if (sq_part) {
        sq = warp_sum(sq);
        if (lane == 0)
          sq_part[(static_cast<int64_t>(b) * g.tiles_m * g.tiles_n + tm * g.tiles_n + tn) * kEpiWarps + ew] = sq;
      }
    }
  }

  __syncthreads();
  if (threadIdx.x == 0 && *abort_flag) {
    // let every TMA copy still in flight land before the CTA exits
    volatile int never = 0;
    for (int s = 0; s < kStages; ++s)
      if (issued[s]) tc::mbar_wait(&full[s], issued[s] - 1, &never);
  }
  __syncthreads();
  // MC: neither CTA exits while the other may still multicast into it or
  // arrive on its barriers
  if (MC) tc::cluster_sync();
  if (warp == 1) {
    __syncwarp();
    tc::fence_after();
    tc::tmem_dealloc(tmem_base, kTmemCols);
  }
}

// ---------------------------------------------------------------------------
// SIMT grouped GEMM (fp32 parity mode): 64 x 64 tiles, 16-wide K chunks,
// 256 threads with 4 x 4 register tiles.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) k_ns_gemm_simt(const __grid_constant__ GemmArgs args) {
  __shared__ float As[16][64];
  __shared__ float Bs[16][64];
  __shared__ float red[8];
  int b, tm, tn;
  const GemmGroup& g = args.g[decode_tile(args, blockIdx.x, b, tm, tn)];
  const int tid = threadIdx.x;
  const int ty = tid >> 4, tx = tid & 15;
  const int m0 = tm * 64, n0 = tn * 64;
  const T* Ab = static_cast<const T*>(g.Abuf) + b * g.a_bs;
  const T* Bb = static_cast<const T*>(g.Bbuf) + b * g.b_bs;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < g.K; k0 += 16) {
    // stage A(i, k) for i in [m0, m0+64), k in [k0, k0+16) as As[k][i]
    for (int e = tid; e < 1024; e += 256) {
      int i, k;
      if (g.a_mn) { k = e >> 6; i = e & 63; } else { i = e >> 4; k = e & 15; }
      const int64_t gi = m0 + i, gk = k0 + k;
      As[k][i] = to_f32(g.a_mn ? Ab[gk * g.a_ld + gi] : Ab[gi * g.a_ld + gk]);
    }
    for (int e = tid; e < 1024; e += 256) {
      int j, k;
      if (g.b_mn) { k = e >> 6; j = e & 63; } else { j = e >> 4; k = e & 15; }
      const int64_t gj = n0 + j, gk = k0 + k;
      Bs[k][j] = to_f32(g.b_mn ? Bb[gk * g.b_ld + gj] : Bb[gj * g.b_ld + gk]);
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      float av[4], bv[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) { av[r] = As[k][ty * 4 + r]; bv[r] = Bs[k][tx * 4 + r]; }
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(av[r], bv[c], acc[r][c]);
    }
    __syncthreads();
  }
  float s = 1.f;
  if (g.scale_pow) {
    const float v = g.inscale[b];
    s = g.scale_pow == 2 ? v * v : v;
  }
  const float ca = g.ca * s, cb = g.cb * s, dg = g.diag * s;
  T* out = static_cast<T*>(g.out) + b * g.out_bs;
  const T* aux = g.aux ? static_cast<const T*>(g.aux) + b * g.aux_bs : nullptr;
  float sq = 0.f;
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int64_t i = m0 + ty * 4 + r;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int64_t j = n0 + tx * 4 + c;
      float x = cb * acc[r][c];
      if (aux) x = fmaf(ca, to_f32(aux[i * g.aux_ld + j]), x);
      if (i == j) x += dg;
      const T y = from_f32<T>(x);
      out[i * g.out_ld + j] = y;
      const float yf = to_f32(y);
      sq += yf * yf;
    }
  }
  if (g.sq_part) {
    sq = block_sum(sq, red);
    if (tid == 0) g.sq_part[static_cast<int64_t>(b) * g.tiles_m * g.tiles_n + tm * g.tiles_n + tn] = sq;
  }
}

// ---------------------------------------------------------------------------
// Prescale 1/(||Psi||_F + eps)
// ---------------------------------------------------------------------------
struct ScaleArgs {
  float* inscale[kMaxGroups];
  const int* mat_ids[kMaxGroups];
  int batch[kMaxGroups];
  int n_groups;
  float eps;
  const int* count;
};
__global__ void k_scale_from_count(const ScaleArgs a) {
  const int gi = blockIdx.x;
  for (int b = threadIdx.x; b < a.batch[gi]; b += blockDim.x) {
    const float m = static_cast<float>(a.count[a.mat_ids[gi][b]]);
    a.inscale[gi][b] = 1.f / (sqrtf(m) + a.eps);
  }
}

template <typename T>
__global__ void k_scale_from_norm(const T* X, int64_t per, float* inscale, float eps) {
  __shared__ double red[32];
  const T* x = X + static_cast<int64_t>(blockIdx.x) * per;
  double s = 0;
  for (int64_t i = threadIdx.x; i < per; i += blockDim.x) {
    const double v = to_f32(x[i]);
    s += v * v;
  }
  s = block_sum(s, red);
  if (threadIdx.x == 0) inscale[blockIdx.x] = static_cast<float>(1.0 / (sqrt(s) + static_cast<double>(eps)));
}

// ---------------------------------------------------------------------------
// Host plan
// ---------------------------------------------------------------------------
struct NSLaunches {
  GemmArgs gram, poly, update;    // per-iteration templates (scale / sq fields patched per run)
  bool mc[3];                     // phase runs on two-CTA clusters sharing B (every tiles_m even)
  CUtensorMap xmap[kMaxGroups][3];  // tensor maps of the X ping-pong buffers
};

// Launch configuration of the two-CTA-cluster GEMM.
static void pair_config(cudaLaunchConfig_t* cfg, cudaLaunchAttribute* attr, int grid, cudaStream_t s) {
  cfg->gridDim = dim3(grid);
  cfg->blockDim = dim3(kTcThreads);
  cfg->dynamicSmemBytes = kTcSmem;
  cfg->stream = s;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg->attrs = attr;
  cfg->numAttrs = 1;
}

NSPlan::~NSPlan() { release(); }

void NSPlan::release() {
  for (void* p : allocs_) cudaFree(p);
  allocs_.clear();
  if (tc_args_host_) {
    delete static_cast<NSLaunches*>(tc_args_host_);
    tc_args_host_ = nullptr;
  }
  groups_.clear();
}

static bool make_map(CUtensorMap* m, void* base, int64_t rows, int64_t cols, int batch,
                     std::string* err) {
  const uint64_t dims[3] = {static_cast<uint64_t>(cols), static_cast<uint64_t>(rows),
                            static_cast<uint64_t>(batch)};
  const uint64_t strides[2] = {static_cast<uint64_t>(cols) * 2, static_cast<uint64_t>(rows * cols) * 2};
  const uint32_t box[3] = {64, 64, 1};
  return driver_encode_tiled(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, base, dims, strides, box, err);
}

cudaError_t NSPlan::init(bool bf16, const std::vector<NSGroupSpec>& specs, std::string* err) {
  release();
  bf16_ = bf16;
  num_sms_ = device_sm_count();
  if (static_cast<int>(specs.size()) > kMaxGroups) {
    if (err) *err = "too many Newton-Schulz shape groups";
    return cudaErrorInvalidValue;
  }
  const int64_t tile_m = bf16 ? 128 : 64;
  for (const NSGroupSpec& sp : specs) {
    NSGroupBuf g;
    g.spec = sp;
    g.tall = sp.rows > sp.cols;
    g.s = std::min(sp.rows, sp.cols);
    g.big = std::max(sp.rows, sp.cols);
    g.elem = bf16 ? 2 : 4;
    if (bf16) {
      g.s_pad = round_up(g.s, 128);
      g.bn_s = (g.s_pad % 256 == 0) ? 256 : 128;
      if (g.tall) {
        // 256: the update of a tall matrix then has an even number of
        // 128-row tiles and can run on two-CTA clusters
        g.big_pad = round_up(g.big, 256);
        g.bn_big = g.bn_s;
      } else {
        g.big_pad = round_up(g.big, 256);
        g.bn_big = 256;
      }
    } else {
      g.s_pad = round_up(g.s, tile_m);
      g.big_pad = round_up(g.big, tile_m);
      g.bn_s = g.bn_big = 64;
    }
    g.rows_pad = g.tall ? g.big_pad : g.s_pad;
    g.cols_pad = g.tall ? g.s_pad : g.big_pad;
    const size_t xbytes = static_cast<size_t>(sp.batch) * g.rows_pad * g.cols_pad * g.elem;
    const size_t abytes = static_cast<size_t>(sp.batch) * g.s_pad * g.s_pad * g.elem;
    // tiles of the update GEMM (its epilogue emits the ||T||^2 partials)
    const int64_t um = g.tall ? g.big_pad : g.s_pad, un = g.tall ? g.s_pad : g.big_pad;
    const int64_t ubn = g.tall ? g.bn_s : g.bn_big;
    const int tiles = static_cast<int>((um / tile_m) * (un / (bf16 ? ubn : 64)));
    g.n_part = tiles * (bf16 ? kEpiWarps : 1);
    void* p;
    for (int i = 0; i < 3; ++i) {
      cudaError_t e = cudaMalloc(&p, xbytes);
      if (e != cudaSuccess) return e;
      allocs_.push_back(p);
      g.X[i] = p;
      cudaMemset(p, 0, xbytes);
    }
    for (void** dst : {&g.A, &g.B}) {
      cudaError_t e = cudaMalloc(&p, abytes);
      if (e != cudaSuccess) return e;
      allocs_.push_back(p);
      *dst = p;
      cudaMemset(p, 0, abytes);
    }
    cudaError_t e = cudaMalloc(&p, sizeof(float) * sp.batch);
    if (e != cudaSuccess) return e;
    allocs_.push_back(p);
    g.inscale = static_cast<float*>(p);
    e = cudaMalloc(&p, sizeof(float) * sp.batch * g.n_part);
    if (e != cudaSuccess) return e;
    allocs_.push_back(p);
    g.sq_part = static_cast<float*>(p);
    groups_.push_back(g);
  }

  // launch descriptors
  NSLaunches* L = new NSLaunches();
  std::memset(L, 0, sizeof(NSLaunches));
  tc_args_host_ = L;
  GemmArgs* phases[3] = {&L->gram, &L->poly, &L->update};
  for (int ph = 0; ph < 3; ++ph) {
    GemmArgs& a = *phases[ph];
    a.n_groups = static_cast<int>(groups_.size());
    int tiles = 0;
    for (size_t gi = 0; gi < groups_.size(); ++gi) {
      NSGroupBuf& gb = groups_[gi];
      GemmGroup& g = a.g[gi];
      const int64_t xs = gb.rows_pad * gb.cols_pad, as = gb.s_pad * gb.s_pad;
      g.batch = gb.spec.batch;
      if (ph == 0) {           // A = X X^T (wide) or X^T X (tall)
        g.M = g.N = static_cast<int>(gb.s_pad);
        g.K = static_cast<int>(gb.big_pad);
        g.a_mn = g.b_mn = gb.tall ? 1 : 0;
        g.BN = bf16 ? gb.bn_s : 64;
        g.a_ld = g.b_ld = gb.cols_pad;
        g.a_bs = g.b_bs = xs;
        g.out_ld = gb.s_pad; g.out_bs = as;
        g.ca = 0.f; g.cb = 1.f;
      } else if (ph == 1) {    // B = b A + c A A   (A symmetric: A A = A A^T)
        g.M = g.N = g.K = static_cast<int>(gb.s_pad);
        g.a_mn = g.b_mn = 0;
        g.BN = bf16 ? gb.bn_s : 64;
        g.Abuf = g.Bbuf = gb.A;
        g.a_ld = g.b_ld = gb.s_pad;
        g.a_bs = g.b_bs = as;
        g.out = gb.B; g.out_ld = gb.s_pad; g.out_bs = as;
        g.aux = gb.A; g.aux_ld = gb.s_pad; g.aux_bs = as;
      } else {                 // X' = a X + B X (wide) or a X + X B (tall)
        g.K = static_cast<int>(gb.s_pad);
        if (!gb.tall) {
          g.M = static_cast<int>(gb.s_pad); g.N = static_cast<int>(gb.big_pad);
          g.a_mn = 0; g.b_mn = 1;
          g.BN = bf16 ? gb.bn_big : 64;
          g.Abuf = gb.B; g.a_ld = gb.s_pad; g.a_bs = as;
          g.b_ld = gb.cols_pad; g.b_bs = xs;          // Bbuf = X_in (set per run)
        } else {
          g.M = static_cast<int>(gb.big_pad); g.N = static_cast<int>(gb.s_pad);
          g.a_mn = 0; g.b_mn = 0;
          g.BN = bf16 ? gb.bn_s : 64;
          g.a_ld = gb.cols_pad; g.a_bs = xs;          // Abuf = X_in (set per run)
          g.Bbuf = gb.B; g.b_ld = gb.s_pad; g.b_bs = as;
        }
        g.out_ld = gb.cols_pad; g.out_bs = xs;
        g.cb = 1.f;
      }
      const int tmM = bf16 ? 128 : 64;
      g.tiles_m = g.M / tmM;
      g.tiles_n = g.N / g.BN;
      // the Gram and polynomial products are symmetric: the tensor-core path
      // computes the tiles on or above the diagonal and mirrors them
      g.sym = (bf16 && ph < 2) ? 1 : 0;
      g.per = tiles_per_matrix(g.tiles_m, g.tiles_n, g.BN, g.sym);
      g.tile_begin = tiles;
      g.b_base = 0;
      tiles += g.batch * g.per;
      if (bf16) {
        // tensor maps: Gram reads X (set per run: one map per X buffer is
        // prepared below); poly reads A; update reads B and X.
        if (ph == 1) {
          if (!make_map(&g.mapA, gb.A, gb.s_pad, gb.s_pad, g.batch, err)) return cudaErrorInvalidValue;
          g.mapB = g.mapA;
        }
        if (ph == 2) {
          CUtensorMap mb;
          if (!make_map(&mb, gb.B, gb.s_pad, gb.s_pad, g.batch, err)) return cudaErrorInvalidValue;
          if (!gb.tall) g.mapA = mb; else g.mapB = mb;
        }
      }
    }
    a.total_tiles = tiles;
    bool cl = bf16;
    for (int gi = 0; gi < a.n_groups; ++gi)
      if (a.g[gi].tiles_m % 2 != 0 || (a.g[gi].BN / 64) % 2 != 0) cl = false;
    L->mc[ph] = cl;
  }
  if (bf16) {
    for (size_t gi = 0; gi < groups_.size(); ++gi) {
      NSGroupBuf& gb = groups_[gi];
      for (int i = 0; i < 3; ++i)
        if (!make_map(&L->xmap[gi][i], gb.X[i], gb.rows_pad, gb.cols_pad, gb.spec.batch, err))
          return cudaErrorInvalidValue;
    }
    cudaError_t e = cudaSuccess;
    for (auto fn : {k_ns_gemm_tc<false>, k_ns_gemm_tc<true>}) {
      e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kTcSmem));
      if (e != cudaSuccess) return e;
    }
    // how many two-CTA clusters fit at once (a GPC with an odd number of
    // usable SMs leaves one of them out); the persistent grid stays within it
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    pair_config(&cfg, attr, 2 * std::max(1, num_sms_ / 2), nullptr);
    int n = 0;
    e = cudaOccupancyMaxActiveClusters(&n, k_ns_gemm_tc<true>, &cfg);
    if (e != cudaSuccess) return e;
    max_pairs_ = n;
    if (n < 1) L->mc[0] = L->mc[1] = L->mc[2] = false;
  }
  return cudaSuccess;
}

// The launch arguments of groups [g0, g0 + cnt) of a prepared grouped
// launch (their tiles are contiguous and keep their order), or with cnt = 1
// of matrices [m0, m1) of group g0 (tiles are matrix-major within a group).
// Returns whether the selection starts and ends on a two-tile cluster unit.
static bool select_groups(GemmArgs& a, int g0, int cnt, int m0, int m1) {
  if (g0 == 0 && cnt == a.n_groups && m0 == 0 && m1 == a.g[0].batch) return true;
  int t0 = a.g[g0].tile_begin;
  int t1 = (g0 + cnt < a.n_groups) ? a.g[g0 + cnt].tile_begin : a.total_tiles;
  for (int j = 0; j < cnt; ++j) {
    a.g[j] = a.g[g0 + j];
    a.g[j].tile_begin -= t0;
  }
  a.n_groups = cnt;
  if (cnt == 1 && (m0 != 0 || m1 != a.g[0].batch)) {
    GemmGroup& g = a.g[0];
    t0 += m0 * g.per;
    t1 = t0 + (m1 - m0) * g.per;
    g.batch = m1 - m0;
    g.b_base = m0;
  }
  a.total_tiles = t1 - t0;
  return (t0 & 1) == 0 && (t1 & 1) == 0;
}

cudaError_t NSPlan::run(int steps, const float coef[3], cudaStream_t s, int* flags, ProfileHook* prof, int g0,
                        int cnt, int m0, int m1) {
  ProfileHook none;
  if (!prof) prof = &none;
  NSLaunches* L = static_cast<NSLaunches*>(tc_args_host_);
  if (!L) return cudaErrorInvalidValue;
  const int ng = static_cast<int>(groups_.size());
  if (cnt < 0) cnt = ng - g0;
  if (g0 < 0 || cnt < 1 || g0 + cnt > ng) return cudaErrorInvalidValue;
  const int batch0 = groups_[g0].spec.batch;
  if (m1 < 0) m1 = batch0;
  if (m0 < 0 || m0 >= m1 || m1 > batch0 || (cnt > 1 && (m0 != 0 || m1 != batch0))) return cudaErrorInvalidValue;
  const float a = coef[0], b = coef[1], c = coef[2];
  for (int it = 0; it < steps; ++it) {
    const int in = (it == 0) ? 0 : ((it % 2 == 1) ? 1 : 2);
    const int out = (it % 2 == 0) ? 1 : 2;
    const bool first = (it == 0), last = (it == steps - 1);
    GemmArgs gram = L->gram, poly = L->poly, upd = L->update;
    gram.flags = poly.flags = upd.flags = flags;
    for (int gi = 0; gi < ng; ++gi) {
      NSGroupBuf& gb = groups_[gi];
      GemmGroup& g0 = gram.g[gi];
      g0.Abuf = g0.Bbuf = gb.X[in];
      g0.out = gb.A;
      g0.scale_pow = first ? 2 : 0;
      g0.inscale = gb.inscale;
      GemmGroup& g1 = poly.g[gi];
      g1.ca = b; g1.cb = c; g1.diag = a;          // C = a I + b A + c A^2
      GemmGroup& g2 = upd.g[gi];
      if (!gb.tall) g2.Bbuf = gb.X[in]; else g2.Abuf = gb.X[in];
      g2.aux = nullptr;
      g2.out = gb.X[out];
      g2.ca = 0.f; g2.cb = 1.f;                   // X' = C X (wide) or X C (tall)
      g2.scale_pow = first ? 1 : 0;
      g2.inscale = gb.inscale;
      g2.sq_part = last ? gb.sq_part : nullptr;
      if (bf16_) {
        g0.mapA = g0.mapB = L->xmap[gi][in];
        if (!gb.tall) g2.mapB = L->xmap[gi][in]; else g2.mapA = L->xmap[gi][in];
      }
    }
    GemmArgs* ph[3] = {&gram, &poly, &upd};
    const int cls[3] = {kProfNsGram, kProfNsPoly, kProfNsUpdate};
    for (int p = 0; p < 3; ++p) {
      const bool units = select_groups(*ph[p], g0, cnt, m0, m1);
      prof->begin(cls[p], s);
      if (bf16_) {
        if (L->mc[p] && units) {
          cudaLaunchConfig_t cfg = {};
          cudaLaunchAttribute attr[1];
          pair_config(&cfg, attr, 2 * std::min(ph[p]->total_tiles / 2, max_pairs_), s);
          cudaError_t le = cudaLaunchKernelEx(&cfg, k_ns_gemm_tc<true>, *ph[p]);
          if (le != cudaSuccess) return le;
        } else {
          const int grid = std::min(ph[p]->total_tiles, num_sms_);
          k_ns_gemm_tc<false><<<grid, kTcThreads, kTcSmem, s>>>(*ph[p]);
        }
      } else {
        k_ns_gemm_simt<float><<<ph[p]->total_tiles, 256, 0, s>>>(*ph[p]);
      }
      cudaError_t e = cudaGetLastError();
      if (e != cudaSuccess) return e;
      prof->end(cls[p], s, 1);
    }
  }
  return cudaSuccess;
}

cudaError_t NSPlan::scale_from_count(const int* count, const int* const* group_mat_ids, float eps,
                                     cudaStream_t s, ProfileHook* prof, int g0, int cnt, int m0, int m1) {
  const int ng = static_cast<int>(groups_.size());
  if (cnt < 0) cnt = ng - g0;
  if (g0 < 0 || cnt < 1 || g0 + cnt > ng) return cudaErrorInvalidValue;
  const int batch0 = groups_[g0].spec.batch;
  if (m1 < 0) m1 = batch0;
  if (m0 < 0 || m0 >= m1 || m1 > batch0 || (cnt > 1 && (m0 != 0 || m1 != batch0))) return cudaErrorInvalidValue;
  ScaleArgs a;
  std::memset(&a, 0, sizeof(a));
  a.n_groups = cnt;
  a.eps = eps;
  a.count = count;
  for (int j = 0; j < cnt; ++j) {
    a.inscale[j] = groups_[g0 + j].inscale + m0;
    a.mat_ids[j] = group_mat_ids[j] + m0;
    a.batch[j] = (cnt == 1) ? m1 - m0 : groups_[g0 + j].spec.batch;
  }
  if (prof) prof->begin(kProfPrescale, s);
  k_scale_from_count<<<a.n_groups, 128, 0, s>>>(a);
  if (prof) prof->end(kProfPrescale, s, 1);
  return cudaGetLastError();
}

cudaError_t NSPlan::scale_from_norm(float eps, cudaStream_t s) {
  for (NSGroupBuf& g : groups_) {
    const int64_t per = g.rows_pad * g.cols_pad;
    if (bf16_) k_scale_from_norm<normpre::bf16><<<g.spec.batch, 512, 0, s>>>(static_cast<const normpre::bf16*>(g.X[0]), per, g.inscale, eps);
    else k_scale_from_norm<float><<<g.spec.batch, 512, 0, s>>>(static_cast<const float*>(g.X[0]), per, g.inscale, eps);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace normpre
