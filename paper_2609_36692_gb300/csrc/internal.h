// Host-side declarations shared by the translation units of libnormpre.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <vector>

namespace normpre {

// Bits of the device status word (see normpre_sync_status).
constexpr int kFlagNonfinite = 1;
constexpr int kFlagNumeric = 2;
constexpr int kFlagTimeout = 4;

constexpr int kMaxBatch = 32;    // matrices served by one normalize/apply launch
constexpr int kMaxGroups = 7;    // shape groups served by one Newton-Schulz GEMM launch (its arguments within 4 KB)

inline int64_t round_up(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

// Kernel classes of the per-phase profile (normpre_profile_read).
enum ProfClass {
  kProfNormalize = 0, kProfNsGram = 1, kProfNsPoly = 2, kProfNsUpdate = 3, kProfApplyG = 4,
  kProfOmega = 5, kProfContract = 6, kProfQR = 7, kProfEig = 8, kProfApplyL = 9,
  kProfPrescale = 10, kProfExactSweeps = 11, kProfExactSelect = 12, kProfClasses = 13
};

// Counts kernel launches and, when enabled, brackets launch groups with CUDA
// events recorded on the launch stream.
class ProfileHook {
 public:
  bool on = false;
  int64_t launches[kProfClasses] = {};
  double ms[kProfClasses] = {};
  void begin(int cls, cudaStream_t s) {
    if (!on) return;
    open_cls_ = cls;
    open_ = take();
    cudaEventRecord(open_, s);
  }
  void end(int cls, cudaStream_t s, int n_launches) {
    launches[cls] += n_launches;
    if (!on || !open_) return;
    cudaEvent_t e = take();
    cudaEventRecord(e, s);
    marks_.push_back({open_cls_, open_, e});
    open_ = nullptr;
  }
  // Waits for the recorded events and folds them into ms[].
  void collect() {
    for (auto& m : marks_) {
      cudaEventSynchronize(m.b);
      float t = 0.f;
      cudaEventElapsedTime(&t, m.a, m.b);
      ms[m.cls] += t;
      pool_.push_back(m.a);
      pool_.push_back(m.b);
    }
    marks_.clear();
  }
  void reset() {
    collect();
    for (int i = 0; i < kProfClasses; ++i) { ms[i] = 0; launches[i] = 0; }
  }
  ~ProfileHook() {
    for (auto& m : marks_) { cudaEventDestroy(m.a); cudaEventDestroy(m.b); }
    for (auto e : pool_) cudaEventDestroy(e);
  }

 private:
  struct Mark { int cls; cudaEvent_t a, b; };
  cudaEvent_t take() {
    if (!pool_.empty()) { cudaEvent_t e = pool_.back(); pool_.pop_back(); return e; }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
  }
  std::vector<Mark> marks_;
  std::vector<cudaEvent_t> pool_;
  cudaEvent_t open_ = nullptr;
  int open_cls_ = 0;
};
inline int64_t cdiv(int64_t x, int64_t m) { return (x + m - 1) / m; }

// ----------------------------------------------------------------------------
// K1: momentum + relaxed tangent + diagonal-Gram normalization (normalize.cu)
// ----------------------------------------------------------------------------
struct NormLaunch {
  int n = 0;                      // matrices in this launch (<= kMaxBatch)
  int64_t rows = 0, cols = 0;     // stored shape
  int g_dtype = 0, w_dtype = 0;   // 0 = f32, 1 = bf16
  int psi_dtype = 0;              // dtype of the written Psi
  const void* G[kMaxBatch] = {};
  float* M[kMaxBatch] = {};       // in: M_{t-1}, out: M_t
  const void* W[kMaxBatch] = {};
  void* psi[kMaxBatch] = {};      // Psi in the stored layout, row stride psi_ld
  int mat_id[kMaxBatch] = {};     // global matrix index (into count[])
  int64_t psi_ld = 0;
  float mu = 0.95f;
  int tangent = 0;                // 0 relaxed (paper), 1 none, 2 strict (Table 5a ablations)
  int* count = nullptr;           // [n_mats] nonzero active rows, accumulated
  int* flags = nullptr;
  // column-active scratch (see normalize_cols_scratch_bytes)
  double* col_part = nullptr;
  float2* col_coef = nullptr;
};
static_assert(sizeof(NormLaunch) + 64 <= 4096, "kernel arguments beyond 4 KB");
cudaError_t launch_normalize_rows(const NormLaunch& a, cudaStream_t s);
// Muon baseline (muon.cu): M = mu M + G written back and copied to a.psi,
// fp64 sums of ||M||^2 of nblk row blocks into part[i * stride + blk] for the
// launch's matrix i; then the prescale 1 / (||M||_F + eps) of `batch` matrices
// whose partials start stride apart.
cudaError_t launch_momentum_copy(const NormLaunch& a, double* part, int nblk, int stride, cudaStream_t s);
cudaError_t launch_muon_prescale(const double* part, int nblk, int stride, int batch, float* inscale, float eps,
                                 cudaStream_t s);
constexpr int kMuonBlocks = 64;   // row blocks per matrix of the Muon momentum pass
cudaError_t launch_normalize_cols(const NormLaunch& a, cudaStream_t s);
// Orientation 3 ("Row+Column/Step"): the columns of a row-normalized Psi
// normalized in place; count[] becomes the number of nonzero columns.
cudaError_t launch_normalize_psi_cols(const NormLaunch& a, cudaStream_t s);
size_t normalize_cols_scratch_bytes(int64_t rows, int64_t cols, int n);
size_t normalize_cols_part_bytes(int64_t rows, int64_t cols, int n);   // col_part share of it

// ----------------------------------------------------------------------------
// K7: NormPre-G apply: W <- W - lr (target * sqrt(mn)/||T|| T + wd W) (apply.cu)
// ----------------------------------------------------------------------------
struct ApplyLaunch {
  int n = 0;
  int64_t rows = 0, cols = 0;
  int w_dtype = 0, t_dtype = 0;
  void* W[kMaxBatch] = {};
  const void* T[kMaxBatch] = {};      // stored layout, row stride t_ld
  const float* sq_part[kMaxBatch] = {};  // n_part partial sums of ||T||^2 per matrix
  float* stats[kMaxBatch] = {};       // optional: receives [k, m', ||T||_F^2]
  int mat_id[kMaxBatch] = {};
  const int* count = nullptr;         // nonzero active rows per matrix (m')
  int k = 0;                          // orientation of this step
  int64_t t_ld = 0;
  int n_part = 0;
  float lr = 0, wd = 0, target = 0.2f;
};
static_assert(sizeof(ApplyLaunch) + 64 <= 4096, "kernel arguments beyond 4 KB");
cudaError_t launch_apply_g(const ApplyLaunch& a, cudaStream_t s);
// Descent-alignment sums <G, T>, ||G||^2, ||T||^2 per matrix into diag[4..6].
struct DiagLaunch {
  int n = 0;
  int64_t rows = 0, cols = 0;
  const void* G[kMaxBatch] = {};
  int g_dtype = 0;
  const void* T[kMaxBatch] = {};      // stored layout, row stride t_ld
  int t_dtype = 0;
  int64_t t_ld = 0;
  double* diag[kMaxBatch] = {};
};
static_assert(sizeof(DiagLaunch) + 64 <= 4096, "kernel arguments beyond 4 KB");
cudaError_t launch_diag_gt(const DiagLaunch& a, cudaStream_t s);

// ----------------------------------------------------------------------------
// Newton-Schulz (ns.cu)
// ----------------------------------------------------------------------------
struct NSGroupSpec {
  int batch = 0;
  int64_t rows = 0, cols = 0;   // stored logical shape of every matrix of the group
};

struct NSGroupBuf {
  NSGroupSpec spec;
  bool tall = false;            // rows > cols: the Gram matrix is X^T X
  int64_t s = 0, big = 0;       // s = min(rows, cols), big = max(rows, cols)
  int64_t s_pad = 0, big_pad = 0;
  int64_t rows_pad = 0, cols_pad = 0;   // padded stored layout of X buffers
  int bn_s = 256, bn_big = 256;         // N tile of the s x s GEMMs / of the update GEMM
  void* X[3] = {};              // [batch][rows_pad][cols_pad]; X[0] receives Psi
  void* A = nullptr;            // [batch][s_pad][s_pad]
  void* B = nullptr;            // [batch][s_pad][s_pad]
  float* inscale = nullptr;     // [batch] 1/(||Psi||_F + eps)
  float* sq_part = nullptr;     // [batch][n_part] partial ||T||_F^2 of the last update
  int n_part = 0;
  size_t elem = 2;              // element size of X, A, B
};

class NSPlan {
 public:
  NSPlan() = default;
  ~NSPlan();
  // Allocates the buffers of every group and prepares launch descriptors.
  // bf16 = true: tcgen05 tensor-core path; false: fp32 SIMT path.
  cudaError_t init(bool bf16, const std::vector<NSGroupSpec>& groups, std::string* err);
  // q iterations of X <- aX + (b A + c A^2) X on X[0] of groups
  // [g0, g0 + cnt) (cnt < 0: every group from g0) -- with cnt = 1, of its
  // matrices [m0, m1) (m1 < 0: to the last) -- with X[0] scaled by inscale[]
  // in the first iteration.  Leaves T in out_index().
  cudaError_t run(int steps, const float coef[3], cudaStream_t s, int* flags,
                  ProfileHook* prof = nullptr, int g0 = 0, int cnt = -1, int m0 = 0, int m1 = -1);
  // Computes inscale[] = 1/(sqrt(count[mat_id]) + eps) for matrices whose Psi
  // rows are unit or zero (Eq. 3), i.e. ||Psi||_F^2 = number of nonzero rows,
  // for the same selection as run(); group_mat_ids[i] (all the group's
  // matrices) belongs to group g0 + i.
  cudaError_t scale_from_count(const int* count, const int* const* group_mat_ids, float eps,
                               cudaStream_t s, ProfileHook* prof = nullptr, int g0 = 0, int cnt = -1,
                               int m0 = 0, int m1 = -1);
  // Computes inscale[] = 1/(||X0||_F + eps) directly from X[0].
  cudaError_t scale_from_norm(float eps, cudaStream_t s);
  static int out_index(int steps) { return (steps % 2 == 1) ? 1 : 2; }
  std::vector<NSGroupBuf>& groups() { return groups_; }
  bool bf16() const { return bf16_; }
  void release();

 private:
  bool bf16_ = true;
  std::vector<NSGroupBuf> groups_;
  std::vector<void*> allocs_;
  void* tc_args_host_ = nullptr;   // prepared kernel arguments (opaque)
  int num_sms_ = 0;
  int max_pairs_ = 0;           // co-resident two-CTA clusters of the tensor-core GEMM
  int* mat_ids_dev_ = nullptr;
};

// ----------------------------------------------------------------------------
// NormPre-L (sketch.cu)
// ----------------------------------------------------------------------------
struct SketchGroup {
  int batch = 0;
  int plan_batch = 0;           // batch the launch shapes are planned for (0: batch); a
                                // slice keeps its group's, so its sums run in the same order
  int64_t rows = 0, cols = 0;   // stored shape
  int w_dtype = 0;
  int64_t ld = 0;               // row stride of Psi (fp32)
  int ell_rows = 0;             // l when rows are active
  int ell_cols = 0;             // l when columns are active
  // device buffers, all [batch][...] contiguous, fp32 unless noted
  float* psi = nullptr;         // [rows][ld]
  float* omega = nullptr;       // [max(rows, cols)][lmax]
  float* y0 = nullptr;          // [max(rows, cols)][lmax]  (Y0 / Z^T / Y / Q scratch)
  float* zt = nullptr;
  float* y = nullptr;
  float* q = nullptr;           // [m_a][l]
  float* bt = nullptr;          // [n_a][l]  B^T = Psi_a^T Q
  float* qk = nullptr;          // [m_a][l]  Q K
  float* kpart = nullptr;       // split-K partials of the contractions
  float* part = nullptr;        // partial Gram sums (fp32, folded with compensation)
  float* kmat = nullptr;        // [l][l] R^{-1} of a CholeskyQR pass, then K = Z_C (Lam_C^{-1/2} - I) Z_C^T
  float* gram = nullptr;        // [l][l] folded Gram of a panel (CholeskyQR, Rayleigh-Ritz)
  float* ritz = nullptr;        // [l]
  float* zvec = nullptr;        // [l][l]
  float* stats = nullptr;       // [8] per matrix
  float* rfac = nullptr;        // CholeskyQR factor of one pass, per matrix
  int lmax = 0;
  int max_part = 0;
  // NORMPRE_L_EXACT (exact.cu): the one-sided block Jacobi work matrix Z
  // [batch][oj_s_pad][oj_lp] (columns contiguous), its column norms, the
  // per-sweep rotation flags, the selected columns and eigenvalues, and all
  // eigenvalues of every matrix (descending)
  float* oj_z = nullptr;
  float* oj_lam = nullptr;      // [batch][oj_s_pad]
  int* oj_flag = nullptr;       // [(sweeps + 1) per matrix]
  int* oj_sel = nullptr;        // [batch][lmax]
  float* oj_sel_lam = nullptr;  // [batch][lmax]
  int64_t oj_s_pad = 0, oj_lp = 0;
  float* eig_all = nullptr;     // [batch][max(rows, cols)]
  // tensor-core contractions: TMA maps of Psi as the K-major (box 32 x 128)
  // and MN-major (box 32 x 32) A operand; tc = false keeps the SIMT kernel
  CUtensorMap psi_map_k, psi_map_mn;
  bool tc = false;
  // NORMPRE_L in NORMPRE_PREC_BF16: Psi stored in bf16 ([rows][ld] bf16 in the
  // same buffer), contracted by contract_bf16.cu (TMA map psi_map_bf, box
  // 64 x 64) against the bf16 hi / lo split of V in vb [batch][vb_bs]
  bool psi_bf16 = false;
  CUtensorMap psi_map_bf;       // box 64 x 64 (contractions)
  CUtensorMap psi_map_apply;    // box 64 x 32 (apply)
  void* vb = nullptr;
  int64_t vb_bs = 0;
};

struct SketchParams {
  int rank = 32, oversample = 8, power_iters = 1;
  int max_sweeps = 30;          // Jacobi sweep cap of the Ritz problem
  int test_stall = 0;           // tests: one CTA of the first contraction skips its first copy
  uint64_t seed = 0;
  int64_t t = 0;
  int k = 0;                    // orientation of this step
  float lr = 0, wd = 0, target = 0.2f;
  bool exact = false;           // NORMPRE_L_EXACT: exact eigenpairs instead of the sketch
  const int* mat_ids_host = nullptr;   // the group's (or slice's) matrix ids, host copy
  double* diag = nullptr;       // [n_mats][8] diagnostics (energies, alignment sums) or null
  const void* const* G = nullptr;      // with diag: the step's gradients (same order as W)
  int g_dtype = 0;
};

cudaError_t sketch_group_alloc(SketchGroup& g, int rank, int oversample, std::vector<void*>& allocs);
// NORMPRE_L_EXACT (exact.cu): the eigensolver workspaces of a group; and the
// exact eigenpairs of every matrix of g into ritz, zvec, kmat, stats, the
// spectral energies (diag) and either q (the eigenvectors) or, when
// *needs_projection is set, the panel y0 whose product Psi_a y0 is q.
cudaError_t exact_group_alloc(SketchGroup& g, std::vector<void*>& allocs);
constexpr int kExactFlagRows = 25;   // per-matrix share of oj_flag (one entry per sweep, and one more)
cudaError_t exact_eigs(SketchGroup& g, const SketchParams& p, int l, const int* mat_ids, const int* count,
                       double* diag, int* flags, cudaStream_t s, ProfileHook* prof, bool* needs_projection);
// Matrices [b0, b1) of a group as a group of their own: the same workspaces
// from its first matrix on, and tensor maps of Psi over those matrices only.
cudaError_t sketch_group_slice(const SketchGroup& g, int b0, int b1, SketchGroup* out);
cudaError_t run_sketch_group(SketchGroup& g, const SketchParams& p, const int* mat_ids,
                             const int* count, void* const* W, int* flags, cudaStream_t s,
                             ProfileHook* prof);

// bf16-Psi sketch contraction (contract_bf16.cu): out = op(Psi) V, op(Psi) =
// Psi (trans = false, K = cols) or Psi^T (trans = true, K = rows), V fp32
// [K][l] (l <= 64), vb the bf16 split scratch (vb_bs elements per matrix,
// at least 2 * round_up(l, 16) * round_up(K, 64)).  With ksplit > 1, out
// receives per-split partials [ksplit][P][l] per matrix (stride out_bs).
struct ContractBf16Launch {
  const CUtensorMap* psi_map;
  bool trans;
  const float* v; int64_t v_bs;
  void* vb; int64_t vb_bs;
  float* out; int64_t out_bs;
  int64_t P, K;
  int l;
  int64_t kchunk;          // multiple of 64
  int ksplit, batch;
  int* flags;
  int stall_first_copy;
};
bool contract_bf16_map(CUtensorMap* map, const void* psi, int64_t rows, int64_t cols, int64_t ld, int batch,
                       int box_rows = 64);
cudaError_t launch_contract_bf16(const ContractBf16Launch& c, cudaStream_t s);

// Records the message returned by normpre_last_error(NULL) on this thread.
void set_thread_error(const std::string& msg);

// Device properties cached per process.
int device_sm_count();
bool driver_encode_tiled(CUtensorMap* map, CUtensorMapDataType dt, uint32_t rank, void* addr,
                         const uint64_t* dims, const uint64_t* strides_bytes, const uint32_t* box,
                         std::string* err);

}  // namespace normpre
