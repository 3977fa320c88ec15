/*
 * normpre.h — C ABI of the GB300 (sm_103a) NormPre optimizer-step library.
 *
 * The library computes the per-matrix update step of NormPre
 * ("Normalize-Then-Precondition", Algorithm 1 of the paper) for a list of 2-D
 * weight matrices on one GPU:
 *
 *   M_t   = mu M_{t-1} + G_t                                  (Sec. 3.1)
 *   k_t   = t mod 2, Wbar = O_k(W), Mbar = O_k(M)             (Sec. 3.1)
 *   x_i   = mbar_i - <mbar_i, wbar_i> wbar_i                  (relaxed tangent momentum, Sec. 3.1)
 *   Psi   = D(X)^{-1} X                                       (Eq. 3, Sec. 2.2)
 *   T     = msign(Psi) by Newton-Schulz        (NormPre-G, Sec. 3.2, App. B)
 *         | (I + U_C (Lam_C^{-1/2} - I) U_C^T) Psi
 *           with (U_C, Lam_C) from the randomized interaction sketch
 *                                              (NormPre-L, Sec. 2.3, Alg. 2)
 *   W    <- W - eta (0.2 O_k^{-1}(T) / RMS(T) + lambda_wd W)  (Sec. 3.1)
 *
 * Conventions shared by every call:
 *   - Matrices are dense, row-major, contiguous, `rows x cols` as stored.
 *   - Device pointers are CUDA device addresses on the current device and must
 *     be 16-byte aligned.  Host pointers are ordinary host addresses.
 *   - A handle belongs to the device that was current at normpre_init; every
 *     call on it makes that device current for its own duration and gives
 *     the caller's current device back before it returns.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *     Calls enqueue work on it and return without synchronizing unless the
 *     description says otherwise.
 *   - Every int-returning call returns a normpre_status.  A text message for
 *     the last failure of a handle is available from normpre_last_error();
 *     failures of calls without a handle are reported by
 *     normpre_last_error(NULL) (thread-local).
 *   - Argument, shape, dtype and alignment errors are found on the host before
 *     any work is enqueued.  Conditions found on the device (non-finite
 *     momentum, numerical breakdown, a bounded wait that gave up) set a flag in
 *     device memory; it is reported by normpre_sync_status().  No kernel traps.
 */
#ifndef NORMPRE_H
#define NORMPRE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct normpre_handle normpre_handle;

/* Variant of the spectral preconditioner (Algorithm 1). */
enum normpre_variant {
  NORMPRE_G = 0,   /* global: T = msign(Psi) by Newton-Schulz (Sec. 3.2) */
  NORMPRE_L = 1,   /* localized: randomized interaction sketch (Alg. 2) */
  NORMPRE_MUON = 2, /* not NormPre: the paper's comparison optimizer Muon (Sec. 2.1, Sec. 4),
                      i.e. Newton-Schulz applied to the momentum itself, with no orientation,
                      tangent or normalization step, and the same RMS-matched update; it
                      shares the Newton-Schulz kernels and serves the latency comparison */
  NORMPRE_L_EXACT = 3 /* localized with exact eigenspace extraction (Sec. 3.2, App. B): the full
                      symmetric eigendecomposition of the interaction matrix Gamma = Psi_a Psi_a^T
                      (m_a x m_a), the up to r largest eigenvalues above one.  Computed without
                      forming Gamma, by a one-sided block Jacobi SVD of Psi (this library's
                      kernels; Gamma's eigenvalues are Psi's squared singular values).  Costs
                      O(sweeps min(m,n)^2 max(m,n)) per matrix: the reference for the sketch and
                      the source of the spectral diagnostics, not a fast path.  The statistics'
                      last slot holds the Jacobi sweeps that still rotated */
};

/* Storage dtypes of caller tensors. */
enum normpre_dtype {
  NORMPRE_F32 = 0,
  NORMPRE_BF16 = 1
};

/* Status codes. */
enum normpre_status {
  NORMPRE_OK = 0,
  NORMPRE_ERR_ARG = 1,        /* null pointer, bad count or bad hyperparameter */
  NORMPRE_ERR_SHAPE = 2,      /* a dimension <= 0 or beyond the supported range */
  NORMPRE_ERR_DTYPE = 3,      /* dtype not supported for that tensor */
  NORMPRE_ERR_ALIGN = 4,      /* a device pointer is not 16-byte aligned */
  NORMPRE_ERR_CUDA = 5,       /* a CUDA runtime call failed (message has the CUDA error) */
  NORMPRE_ERR_NONFINITE = 6,  /* NaN or Inf met in the momentum or weights (device flag) */
  NORMPRE_ERR_NUMERIC = 7,    /* CholeskyQR breakdown or Jacobi sweep cap reached (device flag) */
  NORMPRE_ERR_TIMEOUT = 8,    /* a bounded device-side wait gave up (device flag) */
  NORMPRE_ERR_UNAVAILABLE = 9 /* reserved: no call returns it (NORMPRE_L_EXACT needs no library) */
};

/* Which precision the spectral stage computes in. */
enum normpre_precision {
  NORMPRE_PREC_BF16 = 0,   /* NormPre-G: Psi and the Newton-Schulz operands in bf16 with fp32
                              accumulation on the tensor cores; normalization in fp32.
                              NormPre-L (the sketch; the pure-bf16 setting of the paper's Qwen3
                              runs, App. A): Psi stored in bf16 (rounded once from the fp32
                              normalization), contracted against the bf16 hi + lo split of the
                              fp32 panels with fp32 accumulation; the panels, CholeskyQR,
                              Rayleigh-Ritz and the update stay fp32.  A group with l > 64 keeps
                              an fp32 Psi.  NORMPRE_L_EXACT ignores it (fp32). */
  NORMPRE_PREC_F32 = 1     /* everything in fp32 (parity mode) */
};

/* Hyperparameters (defaults: Table 4 / App. A of the paper). */
typedef struct normpre_config {
  int variant;            /* normpre_variant */
  float momentum;         /* mu = 0.95 */
  float weight_decay;     /* lambda_wd = 0.1 (multiplied by the learning rate) */
  float target_rms;       /* 0.2 (consistent update RMS, Sec. 3.1) */
  int ns_steps;           /* q = 5 Newton-Schulz iterations */
  float ns_coef[3];       /* (a, b, c) of X <- aX + b(XX^T)X + c(XX^T)^2 X; default Muon's
                             quintic (3.4445, -4.7750, 2.0315) */
  float ns_eps;           /* 1e-7: X is divided by ||X||_F + eps before the iteration */
  int rank;               /* r = 32 (interaction rank budget); rank + oversample <= 72 */
  int oversample;         /* o = 8 (the sketch width is l = min(m_a, r + o); l > 64 runs the
                             contractions on the fp32 SIMT kernel instead of the tensor cores) */
  int power_iters;        /* p = 1 */
  uint64_t seed;          /* Philox4x32-10 key of the sketch matrix Omega */
  int precision;          /* normpre_precision */
  int orientation;        /* 0: alternate rows/columns with t (paper); 1: rows only; 2: columns only;
                             3: rows then columns every step (Table 5b "Row+Column/Step", read as:
                             the rows of the row-active tangent momentum normalized, then the columns
                             of the result; preconditioning and update in the row orientation) */
  int tangent;            /* momentum treatment before normalization: 0 relaxed tangent (paper,
                             x_i = m_i - <m_i, w_i> w_i); 1 none (x_i = m_i); 2 strict tangent
                             (x_i = m_i - <m_i, w_i> w_i / ||w_i||^2) -- the Table 5a ablations */
  int diagnostics;        /* 1: every step also accumulates, per matrix, <G, T>, ||G||^2 and
                             ||T||^2 of the raw gradient G and the preconditioned update T (one
                             more read of G and T), for the descent alignment of NORMPRE_BUF_DIAG */
  int jacobi_max_sweeps;  /* NormPre-L: cap on the Jacobi sweeps of the l x l Ritz problem
                             (Alg. 2, eig of Gamma_Q); 0 = default 30, else in [1, 1000].  A step
                             that reaches the cap before converging reports NORMPRE_ERR_NUMERIC */
  int test_stall;         /* tests only, 0 otherwise.  1: in a NormPre-L step, one CTA of the first
                             sketch contraction does not issue its first copy, so its bounded waits
                             give up after about two seconds and the step reports
                             NORMPRE_ERR_TIMEOUT (that step's results are not meaningful; the
                             context stays usable).  It exercises the device-side timeout path */
} normpre_config;

/* Fills `cfg` with the paper's defaults (NormPre-G, bf16 Newton-Schulz). */
void normpre_default_config(normpre_config* cfg);

/*
 * Creates a handle for a fixed list of matrices: the weight matrices W in
 * R^{m x n} that Algorithm 1 updates one by one, with the optimizer's
 * hyperparameters (Table 4, App. A).  The handle holds no optimizer state of
 * the paper's (the momentum M is the caller's), only plans and workspaces.
 *   cfg       hyperparameters (copied).
 *   n_mats    number of matrices (>= 1).
 *   rows/cols host arrays[n_mats] of stored shapes (each >= 1, <= 65536).
 *   w_dtype   host array[n_mats] of normpre_dtype for W (F32 or BF16).
 *   g_dtype   host array[n_mats] of normpre_dtype for G (F32 or BF16).
 *             M is always F32.
 *   out       receives the handle.
 * The handle owns all device workspaces (allocated here with cudaMalloc on the
 * current device) and precomputed launch plans; matrices of equal shape and
 * dtypes are grouped so that one launch serves a whole group.  NORMPRE_G and
 * NORMPRE_MUON serve at most 7 such groups (one grouped Newton-Schulz launch
 * whose arguments stay within 4 KB); more is a SHAPE error.
 * Errors: ARG (null / bad count / bad hyperparameter), SHAPE, DTYPE, CUDA.
 */
int normpre_init(const normpre_config* cfg, int n_mats, const int64_t* rows, const int64_t* cols,
                 const int* w_dtype, const int* g_dtype, normpre_handle** out);

/*
 * One optimizer step (Algorithm 1) for every matrix of the handle.
 *   t        number of steps completed before this one (0 for the first);
 *            selects the orientation k_t = t mod 2 and the sketch stream.
 *   lr       eta_t.
 *   W, G, M  host arrays[n_mats] of DEVICE pointers: W (w_dtype, updated in
 *            place), G (g_dtype, read only), M (fp32 momentum M_{t-1} on
 *            entry, M_t on return).
 *   stream   cudaStream_t.
 * Asynchronous: enqueues the whole step on `stream`.  Workspaces of the
 * handle are reused by the next step, so two steps of one handle must not run
 * concurrently.  Device-detected conditions: see normpre_sync_status().
 * Errors: ARG, ALIGN, CUDA.
 */
int normpre_step(normpre_handle* h, int64_t t, float lr, void* const* W, const void* const* G,
                 void* const* M, void* stream);

/*
 * The same step on HOST buffers: copies W, G and M from host memory to device
 * staging buffers owned by the handle (allocated on the first call), runs
 * normpre_step, copies W and M back, and synchronizes `stream`.  The copies
 * run on two streams of the handle and overlap the step shape group by shape
 * group: a group's normalization starts once its own inputs are in, its M_t
 * goes back while the other groups are preconditioned, its W once its update
 * is done.  Host buffers should be pinned (cudaHostAlloc / torch pin_memory)
 * for full copy speed; they must not be touched until the call returns.
 * Errors: as normpre_step, plus the device-detected conditions of the step.
 */
int normpre_step_host(normpre_handle* h, int64_t t, float lr, void* const* W_host,
                      const void* const* G_host, void* const* M_host, void* stream);

/*
 * Synchronizes `stream`, then reports and clears the device-side flags set
 * since the last call: TIMEOUT, NONFINITE or NUMERIC (the first one found, in
 * that order: a wait that gave up leaves the rest of the step without
 * meaning), else OK.
 */
int normpre_sync_status(normpre_handle* h, void* stream);

/* What normpre_read / normpre_buffer_info can return for one matrix. */
enum normpre_buffer {
  NORMPRE_BUF_PSI = 0,    /* Psi in the stored layout (rows x cols): the normalized update of the
                             last step; bf16 in NORMPRE_PREC_BF16 with NORMPRE_G or NORMPRE_L
                             (l <= 64), else fp32 */
  NORMPRE_BUF_T = 1,      /* NormPre-G: Newton-Schulz result T in the stored layout (rows x cols),
                             same dtype as PSI */
  NORMPRE_BUF_Q = 2,      /* NormPre-L: orthonormal basis Q of the sketch, m_a x l, fp32; a column
                             for a numerically dependent sketch direction (rank(Y) < l) is zero */
  NORMPRE_BUF_RITZ = 3,   /* NormPre-L: all l Ritz values, descending, fp32 (1 x l) */
  NORMPRE_BUF_Z = 4,      /* NormPre-L: Ritz vectors Z (l x l, column j = j-th Ritz value), fp32 */
  NORMPRE_BUF_OMEGA = 5,  /* NormPre-L: sketch matrix Omega of the last step, n_a x l, fp32 */
  NORMPRE_BUF_STATS = 6,  /* 1 x 8 fp32: [k, m', ||T||_F^2, |C|, l, n_a, m_a, s] of the last step,
                             s = Jacobi sweeps of the Ritz problem (NormPre-L) or outer Jacobi
                             sweeps that rotated a column pair (NORMPRE_L_EXACT) */
  NORMPRE_BUF_EIGS = 7,   /* NORMPRE_L_EXACT: all m_a eigenvalues of Gamma, descending (1 x m_a) */
  NORMPRE_BUF_DIAG = 8    /* 1 x 8 fp32 diagnostics of the last step: [E_top, E_remain, E_sub,
                             E_global, cos(G, Phi), ||G||_F, ||T||_F, <G, T>].  The spectral
                             transformation energies sum e_i = (sqrt(lambda_i) - 1)^2 over the
                             eigenvalues of Gamma in C (top, at most r above one), above one but
                             not in C (remain), and in (0, 1) (sub); "nonzero" means lambda_i >
                             1e-6 lambda_max; NaN unless NORMPRE_L_EXACT.  Phi = R_k(T) is the
                             update direction before the learning rate, without weight decay, so
                             cos(G, Phi) = <G, T> / (||G|| ||T||) in the stored layout: the
                             descent alignment of one matrix; NaN unless cfg.diagnostics */
};

/*
 * Shape and dtype of a readable buffer of matrix `mat` (after at least one
 * step).  Errors: ARG (bad mat / what / buffer absent for this variant).
 */
int normpre_buffer_info(const normpre_handle* h, int mat, int what, int64_t* rows, int64_t* cols,
                        int* dtype);

/*
 * Synchronizes the device and copies buffer `what` of matrix `mat` into the
 * host array `dst` (row-major, `capacity_bytes` long).  Intended for tests and
 * diagnostics: the intermediates of the last step as the paper defines them,
 * Psi of Eq. 3, T of Sec. 3.2 (Newton-Schulz), Omega, Q, the Ritz pairs and
 * the selection of Algorithm 2, the eigenvalues of Gamma of the exact
 * extraction (Sec. 3.2), the energies and alignment of App. E.
 * Errors: ARG (too small / absent), CUDA.
 */
int normpre_read(normpre_handle* h, int mat, int what, void* dst, int64_t capacity_bytes);

/*
 * Stand-alone Newton-Schulz (the NormPre-G preconditioner of Sec. 3.2 and
 * App. B; also Muon's orthogonalization):
 *   T_b = NS_q(X_b) for b < batch, X_b rows x cols, contiguous [batch][rows][cols].
 * X and T are device pointers of dtype BF16 when cfg->precision is
 * NORMPRE_PREC_BF16 and F32 otherwise.  X is scaled by 1/(||X_b||_F + eps)
 * first (the scale is computed on the device) and transposed internally when
 * rows > cols.  Uses cfg->ns_steps and cfg->ns_coef.  Allocates its workspace
 * per call and synchronizes `stream` before returning.
 * Errors: ARG, SHAPE, ALIGN, CUDA, TIMEOUT.
 */
int normpre_newton_schulz(const normpre_config* cfg, int batch, int64_t rows, int64_t cols,
                          const void* X, void* T, void* stream);

/*
 * The Gaussian sketch matrix of one matrix and step (Algorithm 2, "sample
 * Omega"), computed by the kernel the NormPre-L step uses, with the random
 * stream it draws from written out for checking:
 *   Omega (n_a x l, row-major, fp32, device): element e = i l + j takes word
 *     e mod 4 of the Philox4x32-10 block (Salmon et al., SC'11) with counter
 *     (e / 4, matrix_id, t lo 32 bits, t hi 32 bits) and key (seed lo, seed
 *     hi); each word x gives the uniform u = ((x >> 9) + 0.5) 2^-23 (exact in
 *     fp32), and the word pairs (0, 1), (2, 3) of a block give two normals by
 *     Box-Muller (sqrt(-2 ln u_a) cos(2 pi u_b), ... sin ...).
 *   words    (optional, NULL to skip; device uint32, n_a x l) the word x of
 *            each element.
 *   uniforms (optional, NULL to skip; device fp32, n_a x l) its uniform u.
 * matrix_id is the matrix's index in the list given to normpre_init (the
 * step's Omega of matrix i at step t equals this call's with matrix_id = i,
 * the same t and the config's seed).  Outputs 4-byte aligned; n_a * l <= 2^32.
 * Asynchronous on `stream`; allocates nothing.
 * Errors (message from normpre_last_error(NULL)): ARG, SHAPE, ALIGN, CUDA.
 */
int normpre_sketch_omega(uint64_t seed, int matrix_id, int64_t t, int64_t n_a, int l, float* omega,
                         uint32_t* words, float* uniforms, void* stream);

/*
 * Per-phase timing of this library's kernels (tests and benchmarks).
 * normpre_profile(h, 1) makes every later step record a pair of CUDA events
 * around each launch group on the step's stream (a few microseconds per step);
 * 0 turns it off.  Kernel launches are always counted.
 */
int normpre_profile(normpre_handle* h, int enable);

/* Kernel classes of normpre_profile_read. */
enum normpre_profile_class {
  NORMPRE_PROF_NORMALIZE = 0,  /* momentum + tangent + normalization (all passes) */
  NORMPRE_PROF_NS_GRAM = 1,    /* Newton-Schulz A = X X^T (or X^T X) */
  NORMPRE_PROF_NS_POLY = 2,    /* Newton-Schulz B = b A + c A^2 */
  NORMPRE_PROF_NS_UPDATE = 3,  /* Newton-Schulz X <- a X + B X (or a X + X B) */
  NORMPRE_PROF_APPLY_G = 4,    /* NormPre-G RMS-matched weight update */
  NORMPRE_PROF_OMEGA = 5,      /* Philox sketch matrix */
  NORMPRE_PROF_CONTRACT = 6,   /* sketch contractions Psi V and Psi^T U */
  NORMPRE_PROF_QR = 7,         /* CholeskyQR passes */
  NORMPRE_PROF_EIG = 8,        /* Rayleigh-Ritz Gram, Jacobi eigensolver, Q K */
  NORMPRE_PROF_APPLY_L = 9,    /* NormPre-L projector apply + weight update */
  NORMPRE_PROF_PRESCALE = 10,  /* Newton-Schulz input scale 1/(sqrt(m') + eps) */
  NORMPRE_PROF_EXACT_SWEEPS = 11,  /* NORMPRE_L_EXACT: the one-sided block Jacobi sweeps over Psi */
  NORMPRE_PROF_EXACT_SELECT = 12,  /* NORMPRE_L_EXACT: eigenvalues, their order, the selection and the
                                      eigenvectors */
  NORMPRE_PROF_CLASSES = 13
};

/*
 * Synchronizes on the recorded events and writes, for each of the first
 * `n_classes` kernel classes, the summed event time in ms (`ms`, zero when
 * profiling was off) and the number of kernel launches (`launches`) since the
 * previous read; then resets both.  Errors: ARG.
 */
int normpre_profile_read(normpre_handle* h, int n_classes, double* ms, int64_t* launches);

/*
 * Allocation-free column-active normalization of ONE matrix (no counterpart
 * in the paper: it exists for callers that cannot allocate device memory when
 * they need this step, such as code running inside a memory-pool or allocator
 * callback, a framework whose allocator must not be re-entered, or a process
 * whose device memory is fully reserved in advance).  It computes what a
 * column-active step (k = 1) of normpre_step computes before the spectral
 * stage, with the same kernels:
 *   M <- mu M + G;  x_j = m_j - <m_j, w_j> w_j per column j;  Psi = x_j / ||x_j||
 * (zero columns give zero columns of Psi).
 *   rows, cols  stored shape (row-major, contiguous), each in [1, 65536] and
 *               rows * cols at most about 87 million (see the scratch limit).
 *   G           device, g_dtype (NORMPRE_F32 or NORMPRE_BF16), read only.
 *   M           device fp32, M_{t-1} on entry, M_t on return.
 *   W           device, w_dtype, read only.
 *   Psi         device fp32 output, rows x cols.
 * Scratch lives in a fixed 8 MiB array in the library's device memory (held
 * by every GPU that loads the library until the process exits); the call
 * performs no cudaMalloc or cudaFree.  Every call shares that array, so calls
 * whose work overlaps on the GPU (on different streams, or concurrently from
 * several host threads on one device) race and give wrong results: order
 * them on one stream.  The first call on each device looks up the array's
 * device address (cudaGetSymbolAddress) with that device current; make that
 * first call before any stream capture.  The address is kept for the life of
 * the process: after cudaDeviceReset (or any other teardown of the device's
 * primary context) it no longer points at the array, so do not call this
 * entry point again in a process that has reset the device.  Asynchronous on `stream`; device-side
 * conditions (non-finite input) are not reported by this entry point.
 * Errors (message from normpre_last_error(NULL)): ARG, SHAPE (including sizes
 * beyond the scratch array), DTYPE, ALIGN, CUDA.
 */
int normpre_normalize_cols_noalloc(int64_t rows, int64_t cols, float mu, const void* G, int g_dtype,
                                   float* M, const void* W, int w_dtype, float* Psi, void* stream);

/* Releases the handle made by normpre_init and every device buffer it owns
 * (the caller's W, G and M, which carry the optimizer's state across the steps
 * of Algorithm 1, are untouched).  NULL is ignored. */
void normpre_free(normpre_handle* h);

/* Message of the last failure of `h` (or of the calling thread when h is NULL). */
const char* normpre_last_error(const normpre_handle* h);

#ifdef __cplusplus
}
#endif
#endif /* NORMPRE_H */
