// C ABI of the NormPre optimizer-step library: handle, shape groups,
// workspaces and the orchestration of one step (Algorithm 1 of the paper).
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <limits>
#include <map>
#include <memory>
#include <string>
#include <tuple>
#include <vector>

#include "../../include/normpre.h"
#include "internal.h"

using namespace normpre;

namespace {

thread_local std::string g_thread_error;

struct MatInfo {
  int64_t rows, cols;
  int w_dtype, g_dtype;
  int group;     // index into groups
  int slot;      // index inside the group
};

struct Group {
  int64_t rows, cols;
  int w_dtype, g_dtype;
  std::vector<int> mats;       // global matrix ids
  int* mat_ids_dev = nullptr;  // device copy of mats
  // NormPre-L
  SketchGroup sk;
};

}  // namespace

void normpre::set_thread_error(const std::string& msg) { g_thread_error = msg; }

struct normpre_handle {
  normpre_config cfg;
  int device = 0;
  int n_mats = 0;
  std::vector<MatInfo> mats;
  std::vector<Group> groups;
  std::vector<void*> allocs;
  int* count = nullptr;        // [n_mats]
  int* flags = nullptr;        // [1]
  float* stats = nullptr;      // [n_mats][8] (NormPre-G)
  double* col_part = nullptr;  // column-active scratch
  float2* col_coef = nullptr;
  double* muon_part = nullptr; // Muon: ||M||^2 partials, [group slot][kMuonBlocks] per group
  double* diag = nullptr;      // [n_mats][8]: spectral energies (exact), alignment sums
  std::unique_ptr<NSPlan> ns;  // NormPre-G and Muon
  int last_k = -1;
  bool stepped = false;
  // host-buffer entry point: device staging per matrix, and the copy streams
  // and per-group events that overlap the copies with the step
  std::vector<void*> stage_w, stage_g, stage_m;
  cudaStream_t h2d = nullptr, d2h = nullptr;
  std::vector<cudaEvent_t> in_ev, norm_ev, upd_ev;   // per unit of work
  cudaEvent_t start_ev = nullptr, out_ev = nullptr;
  ProfileHook prof;
  // NormPre-L: one side stream per shape group so that the groups' sketch
  // pipelines (many small kernels each) run concurrently; joined by events
  std::vector<cudaStream_t> side;
  std::vector<cudaEvent_t> side_fork;   // the group's normalization is done
  std::vector<cudaEvent_t> side_done;
  std::string err;
};

namespace {

int fail(normpre_handle* h, int code, const std::string& msg) {
  if (h) h->err = msg; else g_thread_error = msg;
  return code;
}
int cuda_fail(normpre_handle* h, cudaError_t e, const char* what) {
  return fail(h, NORMPRE_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}
size_t dsize(int dt) { return dt == NORMPRE_BF16 ? 2 : 4; }

// A piece of one step's work: matrices [b0, b1) of shape group g.
struct Unit {
  int g, b0, b1;
};

// How one step's work is cut and ordered, and points of it where a caller
// adds work, called with the unit's index on the stream that runs the unit:
// before its first normalize launch, after its last one (M_t is final), and
// after its update (W is final).
struct StepHooks {
  // the units in the order they are taken (empty: every group whole, in index
  // order)
  std::vector<Unit> units;
  // each unit through all stages before the next one starts; otherwise
  // NormPre-G / Muon run one grouped Newton-Schulz launch over every group,
  // which needs whole groups
  bool per_unit = false;
  virtual ~StepHooks() = default;
  virtual cudaError_t before_normalize(int, cudaStream_t) { return cudaSuccess; }
  virtual cudaError_t after_normalize(int, cudaStream_t) { return cudaSuccess; }
  virtual cudaError_t after_update(int, cudaStream_t) { return cudaSuccess; }
};
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
// Newton-Schulz preconditioning (NormPre-G, Muon) or the localized one (L, L exact)
bool uses_ns(int variant) { return variant == NORMPRE_G || variant == NORMPRE_MUON; }
constexpr int64_t kExactMaxDim = 16384;   // the L-exact selection sorts up to this many eigenvalues in one CTA

int check_config(const normpre_config* c, std::string* msg) {
  if (c->variant != NORMPRE_G && c->variant != NORMPRE_L && c->variant != NORMPRE_MUON &&
      c->variant != NORMPRE_L_EXACT) {
    *msg = "variant must be NORMPRE_G, NORMPRE_L, NORMPRE_MUON or NORMPRE_L_EXACT"; return NORMPRE_ERR_ARG;
  }
  if (c->diagnostics != 0 && c->diagnostics != 1) { *msg = "diagnostics must be 0 or 1"; return NORMPRE_ERR_ARG; }
  if (c->test_stall != 0 && c->test_stall != 1) { *msg = "test_stall must be 0 or 1"; return NORMPRE_ERR_ARG; }
  if (!std::isfinite(c->momentum) || !std::isfinite(c->weight_decay) || !std::isfinite(c->target_rms)) {
    *msg = "momentum, weight_decay and target_rms must be finite"; return NORMPRE_ERR_ARG;
  }
  if (c->precision != NORMPRE_PREC_BF16 && c->precision != NORMPRE_PREC_F32) { *msg = "bad precision"; return NORMPRE_ERR_ARG; }
  if (c->orientation < 0 || c->orientation > 3) { *msg = "orientation must be 0, 1, 2 or 3"; return NORMPRE_ERR_ARG; }
  if (c->tangent < 0 || c->tangent > 2) { *msg = "tangent must be 0, 1 or 2"; return NORMPRE_ERR_ARG; }
  if (c->variant == NORMPRE_L_EXACT) {
    if (c->rank < 1 || c->rank > 72) { *msg = "need 1 <= rank <= 72"; return NORMPRE_ERR_ARG; }
  } else if (uses_ns(c->variant)) {
    if (c->ns_steps < 1 || c->ns_steps > 100) { *msg = "ns_steps must be in [1, 100]"; return NORMPRE_ERR_ARG; }
    if (!std::isfinite(c->ns_coef[0]) || !std::isfinite(c->ns_coef[1]) || !std::isfinite(c->ns_coef[2]) ||
        !(c->ns_eps >= 0.f)) { *msg = "bad Newton-Schulz coefficients or eps"; return NORMPRE_ERR_ARG; }
  } else {
    if (c->rank < 1 || c->oversample < 0 || c->rank + c->oversample > 72) {
      *msg = "need rank >= 1, oversample >= 0 and rank + oversample <= 72"; return NORMPRE_ERR_ARG;
    }
    if (c->power_iters < 0 || c->power_iters > 8) { *msg = "power_iters must be in [0, 8]"; return NORMPRE_ERR_ARG; }
    if (c->jacobi_max_sweeps < 0 || c->jacobi_max_sweeps > 1000) {
      *msg = "jacobi_max_sweeps must be 0 (default) or in [1, 1000]"; return NORMPRE_ERR_ARG;
    }
  }
  return NORMPRE_OK;
}

int orientation_of(const normpre_config& c, int64_t t) {
  if (c.orientation == 1 || c.orientation == 3) return 0;
  if (c.orientation == 2) return 1;
  return static_cast<int>(((t % 2) + 2) % 2);
}

template <typename T>
cudaError_t dalloc(normpre_handle* h, T** p, size_t bytes) {
  void* v = nullptr;
  cudaError_t e = cudaMalloc(&v, bytes);
  if (e != cudaSuccess) return e;
  h->allocs.push_back(v);
  *p = static_cast<T*>(v);
  return cudaMemset(v, 0, bytes);
}

}  // namespace

extern "C" {

void normpre_default_config(normpre_config* c) {
  if (!c) return;
  std::memset(c, 0, sizeof(*c));
  c->variant = NORMPRE_G;
  c->momentum = 0.95f;
  c->weight_decay = 0.1f;
  c->target_rms = 0.2f;
  c->ns_steps = 5;
  c->ns_coef[0] = 3.4445f;
  c->ns_coef[1] = -4.7750f;
  c->ns_coef[2] = 2.0315f;
  c->ns_eps = 1e-7f;
  c->rank = 32;
  c->oversample = 8;
  c->power_iters = 1;
  c->seed = 0;
  c->precision = NORMPRE_PREC_BF16;
  c->orientation = 0;
  c->tangent = 0;
}

const char* normpre_last_error(const normpre_handle* h) {
  return h ? h->err.c_str() : g_thread_error.c_str();
}

namespace {

// Makes the handle's device current for one entry point and gives the caller
// its own current device back on the way out.
class DeviceGuard {
 public:
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev_) == cudaSuccess && prev_ != dev) changed_ = cudaSetDevice(dev) == cudaSuccess;
  }
  ~DeviceGuard() {
    if (changed_) cudaSetDevice(prev_);
  }
  DeviceGuard(const DeviceGuard&) = delete;
  DeviceGuard& operator=(const DeviceGuard&) = delete;

 private:
  int prev_ = 0;
  bool changed_ = false;
};

// Everything a handle holds, on the current device: what normpre_free
// releases, and what a normpre_init that fails part way has created so far.
void release_handle(normpre_handle* h) {
  h->ns.reset();
  for (cudaStream_t st : h->side) cudaStreamDestroy(st);
  for (cudaEvent_t ev : h->side_done) cudaEventDestroy(ev);
  for (cudaEvent_t ev : h->side_fork) cudaEventDestroy(ev);
  for (void* p : h->allocs) cudaFree(p);
  for (auto* v : {&h->stage_w, &h->stage_g, &h->stage_m})
    for (void* p : *v) cudaFree(p);
  for (auto* v : {&h->in_ev, &h->norm_ev, &h->upd_ev})
    for (cudaEvent_t ev : *v) cudaEventDestroy(ev);
  for (cudaEvent_t ev : {h->start_ev, h->out_ev})
    if (ev) cudaEventDestroy(ev);
  for (cudaStream_t st : {h->h2d, h->d2h})
    if (st) cudaStreamDestroy(st);
  delete h;
}

struct HandleRelease {
  void operator()(normpre_handle* h) const { release_handle(h); }
};

}  // namespace

void normpre_free(normpre_handle* h) {
  if (!h) return;
  DeviceGuard device_guard(h->device);
  cudaDeviceSynchronize();
  release_handle(h);
}

int normpre_init(const normpre_config* cfg, int n_mats, const int64_t* rows, const int64_t* cols,
                 const int* w_dtype, const int* g_dtype, normpre_handle** out) {
  if (!cfg || !rows || !cols || !w_dtype || !g_dtype || !out) return fail(nullptr, NORMPRE_ERR_ARG, "null argument");
  *out = nullptr;
  if (n_mats < 1) return fail(nullptr, NORMPRE_ERR_ARG, "n_mats must be >= 1");
  std::string msg;
  int rc = check_config(cfg, &msg);
  if (rc) return fail(nullptr, rc, msg);
  for (int i = 0; i < n_mats; ++i) {
    if (rows[i] < 1 || cols[i] < 1 || rows[i] > 65536 || cols[i] > 65536)
      return fail(nullptr, NORMPRE_ERR_SHAPE, "matrix " + std::to_string(i) + ": each dimension must be in [1, 65536]");
    if (cfg->variant == NORMPRE_L_EXACT && std::max(rows[i], cols[i]) > kExactMaxDim)
      return fail(nullptr, NORMPRE_ERR_SHAPE, "matrix " + std::to_string(i) + ": NORMPRE_L_EXACT supports " +
                  "dimensions up to " + std::to_string(kExactMaxDim));
    if ((w_dtype[i] != NORMPRE_F32 && w_dtype[i] != NORMPRE_BF16) || (g_dtype[i] != NORMPRE_F32 && g_dtype[i] != NORMPRE_BF16))
      return fail(nullptr, NORMPRE_ERR_DTYPE, "matrix " + std::to_string(i) + ": dtype must be NORMPRE_F32 or NORMPRE_BF16");
  }
  // an init that fails part way frees what it has created
  std::unique_ptr<normpre_handle, HandleRelease> h(new normpre_handle());
  h->cfg = *cfg;
  h->n_mats = n_mats;
  cudaError_t e = cudaGetDevice(&h->device);
  if (e != cudaSuccess) return cuda_fail(nullptr, e, "cudaGetDevice");
  // shape groups: equal (rows, cols, w dtype, g dtype)
  std::map<std::tuple<int64_t, int64_t, int, int>, int> key2g;
  h->mats.resize(n_mats);
  for (int i = 0; i < n_mats; ++i) {
    auto key = std::make_tuple(rows[i], cols[i], w_dtype[i], g_dtype[i]);
    auto it = key2g.find(key);
    int gi;
    if (it == key2g.end()) {
      gi = static_cast<int>(h->groups.size());
      key2g[key] = gi;
      Group g;
      g.rows = rows[i]; g.cols = cols[i]; g.w_dtype = w_dtype[i]; g.g_dtype = g_dtype[i];
      h->groups.push_back(g);
    } else {
      gi = it->second;
    }
    h->mats[i] = MatInfo{rows[i], cols[i], w_dtype[i], g_dtype[i], gi, static_cast<int>(h->groups[gi].mats.size())};
    h->groups[gi].mats.push_back(i);
  }
  if (uses_ns(cfg->variant) && h->groups.size() > static_cast<size_t>(kMaxGroups))
    return fail(nullptr, NORMPRE_ERR_SHAPE, "the Newton-Schulz variants support at most " + std::to_string(kMaxGroups) +
                " distinct (shape, dtype) groups per handle");
  normpre_handle* hp = h.get();
  if ((e = dalloc(hp, &h->count, sizeof(int) * n_mats))) return cuda_fail(nullptr, e, "cudaMalloc");
  if ((e = dalloc(hp, &h->flags, sizeof(int) * 4))) return cuda_fail(nullptr, e, "cudaMalloc");
  if ((e = dalloc(hp, &h->stats, sizeof(float) * 8 * n_mats))) return cuda_fail(nullptr, e, "cudaMalloc");
  if ((e = dalloc(hp, &h->diag, sizeof(double) * 8 * n_mats))) return cuda_fail(nullptr, e, "cudaMalloc");
  size_t scratch = 0;
  for (Group& g : h->groups) {
    if ((e = dalloc(hp, &g.mat_ids_dev, sizeof(int) * g.mats.size()))) return cuda_fail(nullptr, e, "cudaMalloc");
    e = cudaMemcpy(g.mat_ids_dev, g.mats.data(), sizeof(int) * g.mats.size(), cudaMemcpyHostToDevice);
    if (e) return cuda_fail(nullptr, e, "cudaMemcpy");
    const int chunk = std::min<int>(kMaxBatch, static_cast<int>(g.mats.size()));
    scratch = std::max(scratch, normalize_cols_scratch_bytes(g.rows, g.cols, chunk));
  }
  if ((e = dalloc(hp, &h->col_part, scratch))) return cuda_fail(nullptr, e, "cudaMalloc");
  {
    int64_t maxc = 1;
    for (Group& g : h->groups) maxc = std::max<int64_t>(maxc, g.cols * std::min<int>(kMaxBatch, static_cast<int>(g.mats.size())));
    if ((e = dalloc(hp, &h->col_coef, sizeof(float2) * maxc))) return cuda_fail(nullptr, e, "cudaMalloc");
  }
  if (cfg->variant == NORMPRE_MUON &&
      (e = dalloc(hp, &h->muon_part, sizeof(double) * kMuonBlocks * n_mats)))
    return cuda_fail(nullptr, e, "cudaMalloc");
  if (uses_ns(cfg->variant)) {
    std::vector<NSGroupSpec> specs;
    for (Group& g : h->groups) specs.push_back(NSGroupSpec{static_cast<int>(g.mats.size()), g.rows, g.cols});
    h->ns.reset(new NSPlan());
    e = h->ns->init(cfg->precision == NORMPRE_PREC_BF16, specs, &msg);
    if (e != cudaSuccess) return fail(nullptr, NORMPRE_ERR_CUDA, "Newton-Schulz plan: " + (msg.empty() ? std::string(cudaGetErrorString(e)) : msg));
  } else {
    for (Group& g : h->groups) {
      g.sk.batch = static_cast<int>(g.mats.size());
      g.sk.rows = g.rows; g.sk.cols = g.cols; g.sk.w_dtype = g.w_dtype;
      g.sk.ld = round_up(g.cols, 8);
      const bool exact = cfg->variant == NORMPRE_L_EXACT;
      // the sketch keeps Psi in bf16 in the bf16 precision mode (where its
      // contraction kernel applies: sketch_group_alloc may clear the flag)
      g.sk.psi_bf16 = !exact && cfg->precision == NORMPRE_PREC_BF16;
      e = sketch_group_alloc(g.sk, cfg->rank, exact ? 0 : cfg->oversample, h->allocs);
      if (e != cudaSuccess) return cuda_fail(nullptr, e, "sketch workspace");
      if (exact) {
        e = exact_group_alloc(g.sk, h->allocs);
        if (e != cudaSuccess) return cuda_fail(nullptr, e, "exact eigensolver workspace");
      }
    }
    if (h->groups.size() > 1) {
      for (size_t gi = 0; gi < h->groups.size(); ++gi) {
        cudaStream_t st;
        cudaEvent_t ev, fev;
        if ((e = cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking))) return cuda_fail(nullptr, e, "cudaStreamCreate");
        h->side.push_back(st);
        if ((e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming))) return cuda_fail(nullptr, e, "cudaEventCreate");
        h->side_done.push_back(ev);
        if ((e = cudaEventCreateWithFlags(&fev, cudaEventDisableTiming))) return cuda_fail(nullptr, e, "cudaEventCreate");
        h->side_fork.push_back(fev);
      }
    }
  }
  e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(nullptr, e, "init");
  *out = h.release();
  return NORMPRE_OK;
}

namespace {

int step_impl(normpre_handle* h, int64_t t, float lr, void* const* W, const void* const* G, void* const* M,
              void* stream, StepHooks& hk) {
  if (!h) return fail(nullptr, NORMPRE_ERR_ARG, "null handle");
  if (!W || !G || !M) return fail(h, NORMPRE_ERR_ARG, "null pointer array");
  if (!std::isfinite(lr)) return fail(h, NORMPRE_ERR_ARG, "lr must be finite");
  for (int i = 0; i < h->n_mats; ++i) {
    if (!W[i] || !G[i] || !M[i]) return fail(h, NORMPRE_ERR_ARG, "matrix " + std::to_string(i) + ": null tensor pointer");
    if (!aligned16(W[i]) || !aligned16(G[i]) || !aligned16(M[i]))
      return fail(h, NORMPRE_ERR_ALIGN, "matrix " + std::to_string(i) + ": tensors must be 16-byte aligned");
  }
  DeviceGuard device_guard(h->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const normpre_config& c = h->cfg;
  const int k = orientation_of(c, t);
  cudaError_t e = cudaMemsetAsync(h->count, 0, sizeof(int) * h->n_mats, s);
  if (e) return cuda_fail(h, e, "cudaMemsetAsync");
  const bool is_muon = (c.variant == NORMPRE_MUON);
  const bool is_g = uses_ns(c.variant);                     // Newton-Schulz preconditioning
  const bool exact = (c.variant == NORMPRE_L_EXACT);
  const bool diag_on = c.diagnostics != 0;
  if ((diag_on || exact) && (e = cudaMemsetAsync(h->diag, 0, sizeof(double) * 8 * h->n_mats, s)))
    return cuda_fail(h, e, "cudaMemsetAsync");
  const bool psi_bf16 = is_g && c.precision == NORMPRE_PREC_BF16;
  // NormPre-L: each group's sketch pipeline runs on its own side stream, from
  // the end of the group's normalization (joined back into `s` at the end),
  // except while per-phase profiling is on, whose event pairs must not overlap
  const bool fork = !is_g && !h->side.empty() && !h->prof.on;

  const int ng = static_cast<int>(h->groups.size());
  std::vector<Unit> units = hk.units;
  if (units.empty())
    for (int gi = 0; gi < ng; ++gi) units.push_back({gi, 0, static_cast<int>(h->groups[gi].mats.size())});
  for (const Unit& u : units) {
    const int B = (u.g >= 0 && u.g < ng) ? static_cast<int>(h->groups[u.g].mats.size()) : 0;
    const bool whole = u.b0 == 0 && u.b1 == B;
    if (u.g < 0 || u.g >= ng || u.b0 < 0 || u.b0 >= u.b1 || u.b1 > B || (!whole && !hk.per_unit))
      return fail(h, NORMPRE_ERR_ARG, "internal: bad unit of work");
  }
  std::vector<int64_t> mslot(ng, 0);   // first Muon partial slot of each group
  for (int gi = 1; gi < ng; ++gi) mslot[gi] = mslot[gi - 1] + static_cast<int64_t>(h->groups[gi - 1].mats.size());

  // (1) momentum + tangent + diagonal-Gram normalization of one unit (Muon:
  //     the momentum alone, copied to the Newton-Schulz input with ||M||^2 sums)
  auto normalize = [&](int ui) -> int {
    const Unit& u = units[ui];
    Group& g = h->groups[u.g];
    char* psi_base;
    int64_t psi_ld, psi_bs;
    if (is_g) {
      NSGroupBuf& nb = h->ns->groups()[u.g];
      psi_base = static_cast<char*>(nb.X[0]);
      psi_ld = nb.cols_pad;
      psi_bs = nb.rows_pad * nb.cols_pad * static_cast<int64_t>(nb.elem);
    } else {
      psi_base = reinterpret_cast<char*>(g.sk.psi);
      psi_ld = g.sk.ld;
      psi_bs = g.rows * g.sk.ld * static_cast<int64_t>(g.sk.psi_bf16 ? 2 : 4);
    }
    cudaError_t e;
    if ((e = hk.before_normalize(ui, s))) return cuda_fail(h, e, "stream wait");
    h->prof.begin(kProfNormalize, s);
    int n_norm = 0;
    for (int c0 = u.b0; c0 < u.b1; c0 += kMaxBatch) {
      NormLaunch a;
      a.n = std::min(kMaxBatch, u.b1 - c0);
      a.rows = g.rows; a.cols = g.cols;
      a.g_dtype = g.g_dtype; a.w_dtype = g.w_dtype;
      a.psi_dtype = (is_g ? psi_bf16 : g.sk.psi_bf16) ? 1 : 0;
      for (int i = 0; i < a.n; ++i) {
        const int mid = g.mats[c0 + i];
        a.G[i] = G[mid]; a.M[i] = static_cast<float*>(M[mid]); a.W[i] = W[mid];
        a.psi[i] = psi_base + static_cast<int64_t>(c0 + i) * psi_bs;
        a.mat_id[i] = mid;
      }
      a.psi_ld = psi_ld;
      a.mu = c.momentum;
      a.tangent = c.tangent;
      a.count = h->count;
      a.flags = h->flags;
      a.col_part = h->col_part;
      a.col_coef = h->col_coef;
      if (is_muon) {
        const int nblk = static_cast<int>(std::min<int64_t>(kMuonBlocks, g.rows));
        e = launch_momentum_copy(a, h->muon_part + (mslot[u.g] + c0) * kMuonBlocks, nblk, kMuonBlocks, s);
        n_norm += 1;
      } else {
        e = (k == 0) ? launch_normalize_rows(a, s) : launch_normalize_cols(a, s);
        n_norm += (k == 0) ? 1 : 3;
        if (!e && c.orientation == 3) {
          e = launch_normalize_psi_cols(a, s);
          n_norm += 3;
        }
      }
      if (e) return cuda_fail(h, e, "normalize launch");
    }
    h->prof.end(kProfNormalize, s, n_norm);
    if (fork && (e = cudaEventRecord(h->side_fork[u.g], s))) return cuda_fail(h, e, "cudaEventRecord");
    if ((e = hk.after_normalize(ui, s))) return cuda_fail(h, e, "copy out");
    return NORMPRE_OK;
  };

  // (2) Newton-Schulz, prescaled by 1/(sqrt(m') + eps) (NormPre-G:
  //     ||Psi||_F^2 = m'), or by 1/(||M||_F + eps) (Muon), on one unit
  //     (ui >= 0) or on every group in one grouped launch per product (ui < 0)
  auto precondition = [&](int ui) -> int {
    const int g0 = ui < 0 ? 0 : units[ui].g, cnt = ui < 0 ? ng : 1;
    const int m0 = ui < 0 ? 0 : units[ui].b0, m1 = ui < 0 ? -1 : units[ui].b1;
    cudaError_t e;
    if (is_muon) {
      h->prof.begin(kProfPrescale, s);
      for (int gi = g0; gi < g0 + cnt; ++gi) {
        Group& g = h->groups[gi];
        const int b0 = ui < 0 ? 0 : m0, b1 = ui < 0 ? static_cast<int>(g.mats.size()) : m1;
        const int nblk = static_cast<int>(std::min<int64_t>(kMuonBlocks, g.rows));
        e = launch_muon_prescale(h->muon_part + (mslot[gi] + b0) * kMuonBlocks, nblk, kMuonBlocks, b1 - b0,
                                 h->ns->groups()[gi].inscale + b0, c.ns_eps, s);
        if (e) return cuda_fail(h, e, "prescale launch");
      }
      h->prof.end(kProfPrescale, s, cnt);
    } else {
      std::vector<const int*> ids;
      for (int gi = g0; gi < g0 + cnt; ++gi) ids.push_back(h->groups[gi].mat_ids_dev);
      e = h->ns->scale_from_count(h->count, ids.data(), c.ns_eps, s, &h->prof, g0, cnt, m0, m1);
      if (e) return cuda_fail(h, e, "prescale launch");
    }
    e = h->ns->run(c.ns_steps, c.ns_coef, s, h->flags, &h->prof, g0, cnt, m0, m1);
    if (e) return cuda_fail(h, e, "Newton-Schulz launch");
    return NORMPRE_OK;
  };

  // (3) RMS-matched update with weight decay of one unit
  auto apply = [&](int ui) -> int {
    const Unit& u = units[ui];
    const int oi = NSPlan::out_index(c.ns_steps);
    Group& g = h->groups[u.g];
    NSGroupBuf& nb = h->ns->groups()[u.g];
    const int64_t xs = nb.rows_pad * nb.cols_pad * static_cast<int64_t>(nb.elem);
    cudaError_t e;
    h->prof.begin(kProfApplyG, s);
    int n_apply = 0;
    for (int c0 = u.b0; c0 < u.b1; c0 += kMaxBatch) {
      ApplyLaunch a;
      a.n = std::min(kMaxBatch, u.b1 - c0);
      a.rows = g.rows; a.cols = g.cols;
      a.w_dtype = g.w_dtype; a.t_dtype = psi_bf16 ? 1 : 0;
      for (int i = 0; i < a.n; ++i) {
        const int mid = g.mats[c0 + i];
        a.W[i] = W[mid];
        a.T[i] = static_cast<char*>(nb.X[oi]) + static_cast<int64_t>(c0 + i) * xs;
        a.sq_part[i] = nb.sq_part + static_cast<int64_t>(c0 + i) * nb.n_part;
        a.stats[i] = h->stats + 8 * mid;
        a.mat_id[i] = mid;
      }
      a.count = h->count;
      a.k = k;
      a.t_ld = nb.cols_pad;
      a.n_part = nb.n_part;
      a.lr = lr; a.wd = c.weight_decay; a.target = c.target_rms;
      if ((e = launch_apply_g(a, s))) return cuda_fail(h, e, "apply launch");
      ++n_apply;
      if (diag_on) {
        // descent alignment: <G, T> with T = the Newton-Schulz output
        DiagLaunch d;
        d.n = a.n; d.rows = g.rows; d.cols = g.cols;
        d.g_dtype = g.g_dtype; d.t_dtype = a.t_dtype; d.t_ld = a.t_ld;
        for (int i = 0; i < a.n; ++i) {
          d.G[i] = G[a.mat_id[i]];
          d.T[i] = a.T[i];
          d.diag[i] = h->diag + 8 * static_cast<int64_t>(a.mat_id[i]);
        }
        if ((e = launch_diag_gt(d, s))) return cuda_fail(h, e, "diagnostics launch");
        ++n_apply;
      }
    }
    h->prof.end(kProfApplyG, s, n_apply);
    if ((e = hk.after_update(ui, s))) return cuda_fail(h, e, "copy out");
    return NORMPRE_OK;
  };

  const int nu = static_cast<int>(units.size());
  int rc;
  if (is_g && hk.per_unit) {
    for (int ui = 0; ui < nu; ++ui)
      if ((rc = normalize(ui)) || (rc = precondition(ui)) || (rc = apply(ui))) return rc;
  } else if (is_g) {
    for (int ui = 0; ui < nu; ++ui)
      if ((rc = normalize(ui))) return rc;
    if ((rc = precondition(-1))) return rc;
    for (int ui = 0; ui < nu; ++ui)
      if ((rc = apply(ui))) return rc;
  } else {
    SketchParams p;
    p.rank = c.rank; p.oversample = c.oversample; p.power_iters = c.power_iters;
    p.seed = c.seed; p.t = t; p.k = k;
    p.max_sweeps = c.jacobi_max_sweeps > 0 ? c.jacobi_max_sweeps : 30;
    p.test_stall = c.test_stall;
    p.lr = lr; p.wd = c.weight_decay; p.target = c.target_rms;
    for (int ui = 0; ui < nu; ++ui) {
      if ((rc = normalize(ui))) return rc;
      const Unit& u = units[ui];
      const int gi = u.g;
      Group& g = h->groups[gi];
      std::vector<void*> wp;
      std::vector<const void*> gp;
      for (int b = u.b0; b < u.b1; ++b) {
        wp.push_back(W[g.mats[b]]);
        gp.push_back(G[g.mats[b]]);
      }
      p.exact = exact;
      p.mat_ids_host = g.mats.data() + u.b0;
      p.diag = (diag_on || exact) ? h->diag : nullptr;
      p.G = diag_on ? gp.data() : nullptr;
      p.g_dtype = g.g_dtype;
      SketchGroup part;
      const bool whole = u.b0 == 0 && u.b1 == static_cast<int>(g.mats.size());
      if (!whole && (e = sketch_group_slice(g.sk, u.b0, u.b1, &part))) return cuda_fail(h, e, "sketch slice");
      cudaStream_t gs = fork ? h->side[gi] : s;
      if (fork && (e = cudaStreamWaitEvent(gs, h->side_fork[gi], 0))) return cuda_fail(h, e, "cudaStreamWaitEvent");
      e = run_sketch_group(whole ? g.sk : part, p, g.mat_ids_dev + u.b0, h->count, wp.data(), h->flags, gs, &h->prof);
      if (e) return cuda_fail(h, e, "sketch launch");
      if ((e = hk.after_update(ui, gs))) return cuda_fail(h, e, "copy out");
      if (fork && (e = cudaEventRecord(h->side_done[gi], gs))) return cuda_fail(h, e, "cudaEventRecord");
    }
    if (fork)
      for (int gi = 0; gi < ng; ++gi)
        if ((e = cudaStreamWaitEvent(s, h->side_done[gi], 0))) return cuda_fail(h, e, "cudaStreamWaitEvent");
  }
  h->last_k = k;
  h->stepped = true;
  return NORMPRE_OK;
}

}  // namespace

int normpre_step(normpre_handle* h, int64_t t, float lr, void* const* W, const void* const* G, void* const* M,
                 void* stream) {
  StepHooks none;
  return step_impl(h, t, lr, W, G, M, stream, none);
}

int normpre_profile(normpre_handle* h, int enable) {
  if (!h) return fail(nullptr, NORMPRE_ERR_ARG, "null handle");
  h->prof.collect();
  h->prof.on = enable != 0;
  return NORMPRE_OK;
}

int normpre_profile_read(normpre_handle* h, int n_classes, double* ms, int64_t* launches) {
  if (!h) return fail(nullptr, NORMPRE_ERR_ARG, "null handle");
  if (n_classes < 0 || (n_classes > 0 && (!ms || !launches))) return fail(h, NORMPRE_ERR_ARG, "bad output arrays");
  DeviceGuard device_guard(h->device);
  h->prof.collect();
  for (int i = 0; i < n_classes; ++i) {
    ms[i] = i < kProfClasses ? h->prof.ms[i] : 0.0;
    launches[i] = i < kProfClasses ? h->prof.launches[i] : 0;
  }
  h->prof.reset();
  return NORMPRE_OK;
}

int normpre_sync_status(normpre_handle* h, void* stream) {
  if (!h) return fail(nullptr, NORMPRE_ERR_ARG, "null handle");
  DeviceGuard device_guard(h->device);
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e) return cuda_fail(h, e, "cudaStreamSynchronize");
  int flags = 0;
  e = cudaMemcpy(&flags, h->flags, sizeof(int), cudaMemcpyDeviceToHost);
  if (e) return cuda_fail(h, e, "cudaMemcpy");
  if (flags) {
    e = cudaMemset(h->flags, 0, sizeof(int));
    if (e) return cuda_fail(h, e, "cudaMemset");
  }
  // a wait that gave up leaves the rest of the step without meaning: first
  if (flags & kFlagTimeout) return fail(h, NORMPRE_ERR_TIMEOUT, "a bounded device wait gave up");
  if (flags & kFlagNonfinite) return fail(h, NORMPRE_ERR_NONFINITE, "non-finite value in the momentum or the weights");
  if (flags & kFlagNumeric) return fail(h, NORMPRE_ERR_NUMERIC, "CholeskyQR breakdown or Jacobi sweep cap reached");
  return NORMPRE_OK;
}

namespace {

// Copies of the host-buffer step, overlapped with it.  The step is cut into
// units of at most kHostUnitBytes of input, largest groups first; the host-to-device stream brings in each unit's W, G,
// M (one event per unit, which the unit's normalize waits on), and one
// device-to-host stream sends each unit's M_t back once its normalize is done
// and its W once its update is done.  A small unit then starts the outgoing
// copies early, and the step ends on a small unit's work.
constexpr int64_t kHostUnitBytes = 256ll << 20;

struct HostPipe : StepHooks {
  normpre_handle* h;
  void* const* W_host;
  void* const* M_host;
  cudaError_t copy_out(int ui, cudaStream_t s, std::vector<cudaEvent_t>& ev, void* const* host,
                       const std::vector<void*>& stage, bool weights) {
    const Unit& u = units[ui];
    cudaError_t e = cudaEventRecord(ev[ui], s);
    if (!e) e = cudaStreamWaitEvent(h->d2h, ev[ui], 0);
    for (int b = u.b0; b < u.b1 && !e; ++b) {
      const int mid = h->groups[u.g].mats[b];
      const MatInfo& m = h->mats[mid];
      const size_t bytes = static_cast<size_t>(m.rows * m.cols) * (weights ? dsize(m.w_dtype) : 4);
      e = cudaMemcpyAsync(host[mid], stage[mid], bytes, cudaMemcpyDeviceToHost, h->d2h);
    }
    return e;
  }
  cudaError_t before_normalize(int ui, cudaStream_t s) override { return cudaStreamWaitEvent(s, h->in_ev[ui], 0); }
  cudaError_t after_normalize(int ui, cudaStream_t s) override {
    return copy_out(ui, s, h->norm_ev, M_host, h->stage_m, false);
  }
  cudaError_t after_update(int ui, cudaStream_t s) override {
    return copy_out(ui, s, h->upd_ev, W_host, h->stage_w, true);
  }
};

// The staging buffers (indexed by matrix), copy streams and step events of
// the host-buffer entry point; all or nothing, so that a retry after a failed
// allocation starts from empty vectors.
void host_pipe_release(normpre_handle* h) {
  for (auto* v : {&h->stage_w, &h->stage_g, &h->stage_m}) {
    for (void* p : *v) cudaFree(p);
    v->clear();
  }
  for (cudaEvent_t* ev : {&h->start_ev, &h->out_ev})
    if (*ev) { cudaEventDestroy(*ev); *ev = nullptr; }
  for (cudaStream_t* st : {&h->h2d, &h->d2h})
    if (*st) { cudaStreamDestroy(*st); *st = nullptr; }
}

cudaError_t host_pipe_alloc_all(normpre_handle* h) {
  cudaError_t e;
  for (int i = 0; i < h->n_mats; ++i) {
    const MatInfo& m = h->mats[i];
    const size_t n = static_cast<size_t>(m.rows * m.cols);
    void *pw = nullptr, *pg = nullptr, *pm = nullptr;
    if ((e = cudaMalloc(&pw, n * dsize(m.w_dtype)))) return e;
    h->stage_w.push_back(pw);
    if ((e = cudaMalloc(&pg, n * dsize(m.g_dtype)))) return e;
    h->stage_g.push_back(pg);
    if ((e = cudaMalloc(&pm, n * 4))) return e;
    h->stage_m.push_back(pm);
  }
  if ((e = cudaStreamCreateWithFlags(&h->h2d, cudaStreamNonBlocking))) return e;
  if ((e = cudaStreamCreateWithFlags(&h->d2h, cudaStreamNonBlocking))) return e;
  if ((e = cudaEventCreateWithFlags(&h->start_ev, cudaEventDisableTiming))) return e;
  return cudaEventCreateWithFlags(&h->out_ev, cudaEventDisableTiming);
}

cudaError_t host_pipe_alloc(normpre_handle* h) {
  const cudaError_t e = host_pipe_alloc_all(h);
  if (e != cudaSuccess) host_pipe_release(h);
  return e;
}

// The units of a host-buffer step, largest groups first.
std::vector<Unit> host_units(const normpre_handle* h) {
  std::vector<std::pair<int64_t, int>> by_size;
  for (size_t gi = 0; gi < h->groups.size(); ++gi) {
    const Group& g = h->groups[gi];
    by_size.push_back({-g.rows * g.cols * static_cast<int64_t>(g.mats.size()), static_cast<int>(gi)});
  }
  std::stable_sort(by_size.begin(), by_size.end());
  std::vector<Unit> units;
  for (auto& sz : by_size) {
    const Group& g = h->groups[sz.second];
    const int B = static_cast<int>(g.mats.size());
    const int64_t bytes = g.rows * g.cols * static_cast<int64_t>(dsize(g.w_dtype) + dsize(g.g_dtype) + 4) * B;
    const int pieces = static_cast<int>(std::min<int64_t>(B, cdiv(bytes, kHostUnitBytes)));
    for (int p = 0; p < pieces; ++p)
      units.push_back({sz.second, static_cast<int>(static_cast<int64_t>(B) * p / pieces),
                       static_cast<int>(static_cast<int64_t>(B) * (p + 1) / pieces)});
  }
  return units;
}

}  // namespace

int normpre_step_host(normpre_handle* h, int64_t t, float lr, void* const* W_host, const void* const* G_host,
                      void* const* M_host, void* stream) {
  if (!h) return fail(nullptr, NORMPRE_ERR_ARG, "null handle");
  if (!W_host || !G_host || !M_host) return fail(h, NORMPRE_ERR_ARG, "null pointer array");
  for (int i = 0; i < h->n_mats; ++i)
    if (!W_host[i] || !G_host[i] || !M_host[i]) return fail(h, NORMPRE_ERR_ARG, "null host tensor pointer");
  DeviceGuard device_guard(h->device);
  cudaError_t e;
  if (!h->h2d && (e = host_pipe_alloc(h))) return cuda_fail(h, e, "host-buffer staging");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  HostPipe pipe;
  pipe.h = h;
  pipe.W_host = W_host;
  pipe.M_host = M_host;
  pipe.units = host_units(h);
  pipe.per_unit = true;
  for (auto* v : {&h->in_ev, &h->norm_ev, &h->upd_ev})
    while (v->size() < pipe.units.size()) {
      cudaEvent_t ev;
      if ((e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming))) return cuda_fail(h, e, "cudaEventCreate");
      v->push_back(ev);
    }
  // the copies start after the work already queued on `s`
  if ((e = cudaEventRecord(h->start_ev, s))) return cuda_fail(h, e, "cudaEventRecord");
  if ((e = cudaStreamWaitEvent(h->h2d, h->start_ev, 0)) || (e = cudaStreamWaitEvent(h->d2h, h->start_ev, 0)))
    return cuda_fail(h, e, "cudaStreamWaitEvent");
  for (size_t ui = 0; ui < pipe.units.size(); ++ui) {
    const Unit& u = pipe.units[ui];
    for (int b = u.b0; b < u.b1; ++b) {
      const int mid = h->groups[u.g].mats[b];
      const MatInfo& m = h->mats[mid];
      const size_t n = static_cast<size_t>(m.rows * m.cols);
      if ((e = cudaMemcpyAsync(h->stage_w[mid], W_host[mid], n * dsize(m.w_dtype), cudaMemcpyHostToDevice, h->h2d)) ||
          (e = cudaMemcpyAsync(h->stage_g[mid], G_host[mid], n * dsize(m.g_dtype), cudaMemcpyHostToDevice, h->h2d)) ||
          (e = cudaMemcpyAsync(h->stage_m[mid], M_host[mid], n * 4, cudaMemcpyHostToDevice, h->h2d)))
        return cuda_fail(h, e, "H2D");
    }
    if ((e = cudaEventRecord(h->in_ev[ui], h->h2d))) return cuda_fail(h, e, "cudaEventRecord");
  }
  int rc = step_impl(h, t, lr, h->stage_w.data(), const_cast<const void* const*>(h->stage_g.data()),
                     h->stage_m.data(), stream, pipe);
  if (rc) {
    cudaStreamSynchronize(h->h2d);
    cudaStreamSynchronize(h->d2h);
    return rc;
  }
  // `s` (and the caller) sees the step complete once the last copy is back
  if ((e = cudaEventRecord(h->out_ev, h->d2h)) || (e = cudaStreamWaitEvent(s, h->out_ev, 0)))
    return cuda_fail(h, e, "cudaEventRecord");
  return normpre_sync_status(h, stream);
}

int normpre_buffer_info(const normpre_handle* h, int mat, int what, int64_t* rows, int64_t* cols, int* dtype) {
  normpre_handle* hh = const_cast<normpre_handle*>(h);
  if (!h) return fail(nullptr, NORMPRE_ERR_ARG, "null handle");
  if (mat < 0 || mat >= h->n_mats) return fail(hh, NORMPRE_ERR_ARG, "bad matrix index");
  if (!h->stepped) return fail(hh, NORMPRE_ERR_ARG, "no step has run yet");
  const MatInfo& m = h->mats[mat];
  const bool is_g = uses_ns(h->cfg.variant);
  const bool rows_active = h->last_k == 0;
  const int64_t m_a = rows_active ? m.rows : m.cols, n_a = rows_active ? m.cols : m.rows;
  int64_t r = 0, c = 0;
  int dt = NORMPRE_F32;
  switch (what) {
    case NORMPRE_BUF_PSI:
      r = m.rows; c = m.cols;
      dt = ((is_g && h->cfg.precision == NORMPRE_PREC_BF16) || (!is_g && h->groups[m.group].sk.psi_bf16))
               ? NORMPRE_BF16 : NORMPRE_F32;
      break;
    case NORMPRE_BUF_T:
      if (!is_g) return fail(hh, NORMPRE_ERR_ARG, "T is kept only for NormPre-G");
      r = m.rows; c = m.cols;
      dt = h->cfg.precision == NORMPRE_PREC_BF16 ? NORMPRE_BF16 : NORMPRE_F32;
      break;
    case NORMPRE_BUF_Q: case NORMPRE_BUF_RITZ: case NORMPRE_BUF_Z: case NORMPRE_BUF_OMEGA: {
      if (is_g) return fail(hh, NORMPRE_ERR_ARG, "sketch buffers exist only for NormPre-L");
      if (what == NORMPRE_BUF_OMEGA && h->cfg.variant == NORMPRE_L_EXACT)
        return fail(hh, NORMPRE_ERR_ARG, "NORMPRE_L_EXACT draws no sketch matrix");
      const SketchGroup& sk = h->groups[m.group].sk;
      const int64_t l = rows_active ? sk.ell_rows : sk.ell_cols;
      if (what == NORMPRE_BUF_Q) { r = m_a; c = l; }
      if (what == NORMPRE_BUF_RITZ) { r = 1; c = l; }
      if (what == NORMPRE_BUF_Z) { r = l; c = l; }
      if (what == NORMPRE_BUF_OMEGA) { r = n_a; c = l; }
      break;
    }
    case NORMPRE_BUF_STATS:
      r = 1; c = 8;
      break;
    case NORMPRE_BUF_EIGS:
      if (h->cfg.variant != NORMPRE_L_EXACT) return fail(hh, NORMPRE_ERR_ARG, "all eigenvalues exist only for NORMPRE_L_EXACT");
      r = 1; c = m_a;
      break;
    case NORMPRE_BUF_DIAG:
      r = 1; c = 8;
      break;
    default:
      return fail(hh, NORMPRE_ERR_ARG, "unknown buffer");
  }
  if (rows) *rows = r;
  if (cols) *cols = c;
  if (dtype) *dtype = dt;
  return NORMPRE_OK;
}

int normpre_read(normpre_handle* h, int mat, int what, void* dst, int64_t capacity_bytes) {
  if (!h) return fail(nullptr, NORMPRE_ERR_ARG, "null handle");
  if (!dst) return fail(h, NORMPRE_ERR_ARG, "null destination");
  int64_t r, c;
  int dt;
  int rc = normpre_buffer_info(h, mat, what, &r, &c, &dt);
  if (rc) return rc;
  const size_t el = dsize(dt);
  if (capacity_bytes < static_cast<int64_t>(r * c * el)) return fail(h, NORMPRE_ERR_ARG, "destination too small");
  DeviceGuard device_guard(h->device);
  cudaError_t e = cudaDeviceSynchronize();
  if (e) return cuda_fail(h, e, "cudaDeviceSynchronize");
  const MatInfo& m = h->mats[mat];
  const Group& g = h->groups[m.group];
  const bool is_g = uses_ns(h->cfg.variant);
  if (what == NORMPRE_BUF_DIAG) {
    // fp64 sums on the device -> [E_top, E_remain, E_sub, E_global, cos, ||G||, ||T||, <G, T>]
    double d[8];
    e = cudaMemcpy(d, h->diag + 8 * static_cast<int64_t>(mat), sizeof(d), cudaMemcpyDeviceToHost);
    if (e) return cuda_fail(h, e, "cudaMemcpy");
    const float nan = std::numeric_limits<float>::quiet_NaN();
    float out[8];
    const bool ex = h->cfg.variant == NORMPRE_L_EXACT, al = h->cfg.diagnostics != 0;
    for (int i = 0; i < 4; ++i) out[i] = ex ? static_cast<float>(d[i]) : nan;
    const double gn = std::sqrt(d[5]), tn = std::sqrt(d[6]);
    out[4] = al ? ((gn > 0 && tn > 0) ? static_cast<float>(d[4] / (gn * tn)) : 0.f) : nan;
    out[5] = al ? static_cast<float>(gn) : nan;
    out[6] = al ? static_cast<float>(tn) : nan;
    out[7] = al ? static_cast<float>(d[4]) : nan;
    std::memcpy(dst, out, sizeof(out));
    return NORMPRE_OK;
  }
  const void* src = nullptr;
  int64_t src_ld = c;
  if (what == NORMPRE_BUF_PSI || what == NORMPRE_BUF_T) {
    if (is_g) {
      NSGroupBuf& nb = h->ns->groups()[m.group];
      const int idx = (what == NORMPRE_BUF_PSI) ? 0 : NSPlan::out_index(h->cfg.ns_steps);
      src = static_cast<char*>(nb.X[idx]) + static_cast<int64_t>(m.slot) * nb.rows_pad * nb.cols_pad * nb.elem;
      src_ld = nb.cols_pad;
    } else {
      src = g.sk.psi_bf16 ? static_cast<const void*>(reinterpret_cast<const uint16_t*>(g.sk.psi) +
                                                      static_cast<int64_t>(m.slot) * g.rows * g.sk.ld)
                          : static_cast<const void*>(g.sk.psi + static_cast<int64_t>(m.slot) * g.rows * g.sk.ld);
      src_ld = g.sk.ld;
    }
  } else if (what == NORMPRE_BUF_STATS) {
    src = is_g ? h->stats + 8 * mat : g.sk.stats + 8 * m.slot;
  } else {
    const SketchGroup& sk = g.sk;
    const int64_t vbs = std::max(sk.rows, sk.cols) * sk.lmax;
    const int64_t sq = static_cast<int64_t>(sk.lmax) * sk.lmax;
    if (what == NORMPRE_BUF_Q) src = sk.q + m.slot * vbs;
    if (what == NORMPRE_BUF_OMEGA) src = sk.omega + m.slot * vbs;
    if (what == NORMPRE_BUF_RITZ) src = sk.ritz + m.slot * sk.lmax;
    if (what == NORMPRE_BUF_Z) src = sk.zvec + m.slot * sq;
    if (what == NORMPRE_BUF_EIGS) src = sk.eig_all + m.slot * std::max(sk.rows, sk.cols);
  }
  e = cudaMemcpy2D(dst, c * el, src, src_ld * el, c * el, r, cudaMemcpyDeviceToHost);
  if (e) return cuda_fail(h, e, "cudaMemcpy2D");
  return NORMPRE_OK;
}

int normpre_newton_schulz(const normpre_config* cfg, int batch, int64_t rows, int64_t cols, const void* X, void* T,
                          void* stream) {
  if (!cfg || !X || !T) return fail(nullptr, NORMPRE_ERR_ARG, "null argument");
  if (batch < 1) return fail(nullptr, NORMPRE_ERR_ARG, "batch must be >= 1");
  if (rows < 1 || cols < 1 || rows > 65536 || cols > 65536) return fail(nullptr, NORMPRE_ERR_SHAPE, "dimensions must be in [1, 65536]");
  if (cfg->ns_steps < 1 || cfg->ns_steps > 100) return fail(nullptr, NORMPRE_ERR_ARG, "ns_steps must be in [1, 100]");
  if (cfg->precision != NORMPRE_PREC_BF16 && cfg->precision != NORMPRE_PREC_F32) return fail(nullptr, NORMPRE_ERR_ARG, "bad precision");
  if (!aligned16(X) || !aligned16(T)) return fail(nullptr, NORMPRE_ERR_ALIGN, "X and T must be 16-byte aligned");
  const bool bf = cfg->precision == NORMPRE_PREC_BF16;
  const size_t el = bf ? 2 : 4;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  NSPlan plan;
  std::string msg;
  cudaError_t e = plan.init(bf, {NSGroupSpec{batch, rows, cols}}, &msg);
  if (e) return fail(nullptr, NORMPRE_ERR_CUDA, "Newton-Schulz plan: " + (msg.empty() ? std::string(cudaGetErrorString(e)) : msg));
  int* flags = nullptr;
  if ((e = cudaMalloc(&flags, sizeof(int)))) return cuda_fail(nullptr, e, "cudaMalloc");
  cudaMemsetAsync(flags, 0, sizeof(int), s);
  NSGroupBuf& g = plan.groups()[0];
  const int64_t xs = g.rows_pad * g.cols_pad;
  for (int b = 0; b < batch && !e; ++b)
    e = cudaMemcpy2DAsync(static_cast<char*>(g.X[0]) + b * xs * el, g.cols_pad * el,
                          static_cast<const char*>(X) + b * rows * cols * el, cols * el, cols * el, rows,
                          cudaMemcpyDeviceToDevice, s);
  if (!e) e = plan.scale_from_norm(cfg->ns_eps, s);
  if (!e) e = plan.run(cfg->ns_steps, cfg->ns_coef, s, flags);
  const int oi = NSPlan::out_index(cfg->ns_steps);
  for (int b = 0; b < batch && !e; ++b)
    e = cudaMemcpy2DAsync(static_cast<char*>(T) + b * rows * cols * el, cols * el,
                          static_cast<char*>(g.X[oi]) + b * xs * el, g.cols_pad * el, cols * el, rows,
                          cudaMemcpyDeviceToDevice, s);
  if (!e) e = cudaStreamSynchronize(s);
  int hf = 0;
  if (!e) e = cudaMemcpy(&hf, flags, sizeof(int), cudaMemcpyDeviceToHost);
  cudaFree(flags);
  if (e) return cuda_fail(nullptr, e, "Newton-Schulz");
  if (hf & kFlagTimeout) return fail(nullptr, NORMPRE_ERR_TIMEOUT, "a bounded device wait gave up");
  return NORMPRE_OK;
}

}  // extern "C"
