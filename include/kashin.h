/*
 * libkashin -- C ABI of the GB300 (sm_103a) Kashin-DCT decomposition and 2-bit coder.
 *
 * The method (arxiv 2609.11687, "Structured Transforms for Low-Overhead
 * Quantization of Language Models"):
 *   - every weight vector x of length n (a column of the paper's n x m matrix W,
 *     App. C) is decomposed by Algorithm 1 (Greedy Algorithm with Alternating
 *     Updates) into  x = u + P vhat + r,  P = IDCT o T_eps o DCT  (Sec. 3.1), with
 *     the orthonormal DCT-II and one sign set eps in {+-1}^n per matrix drawn from
 *     a seed (App. C);
 *   - each factor is coded to 2 bits with the closed-form centres +-c1 +-c2
 *     (u, from the two u-steps of block 0) and +-d1 +-d2 (vhat, from the two
 *     vhat-steps of block 0), nearest centre, ties to the lower code (Sec. 2.1);
 *   - the dequantised weight is  W_hat = U_q + P V_q  (App. C, dense
 *     re-materialisation at load time).
 *
 * Conventions shared by every call
 * --------------------------------
 *  n       vector length (the paper's N: rows of W, input features).
 *  m       number of vectors (the paper's M: columns of W, output channels).
 *  layout  KD_VEC_ROWS:    vector j is w[j*ld + i], i < n  (row-major m x ld, ld >= n;
 *                          the nn.Linear weight layout [out, in]).
 *          KD_VEC_COLUMNS: vector j is w[i*ld + j], i < n  (row-major n x ld, ld >= m;
 *                          the paper's N x M matrix).
 *  sign seed   eps_j = +1, or -1 where bit 63 of SplitMix64(seed + (j+1)*0x9E3779B97F4A7C15)
 *              is set (SplitMix64: Steele, Lea & Flood, OOPSLA 2014).  The paper
 *              does not name its generator; this is the library's fixed choice.
 *  Pointers    every array argument is DEVICE memory owned by the caller unless
 *              it is named *_host.  The library allocates nothing per call.
 *  stream      a cudaStream_t passed as void* (NULL = legacy default stream).
 *              Calls validate their arguments synchronously, then only enqueue
 *              work on the stream and return.
 *  Errors      argument / size / plan problems are returned synchronously and
 *              nothing is enqueued; a failed launch returns KD_ERR_CUDA; a
 *              non-finite input value, or a bounded wait that expired (the CTA
 *              then leaves its remaining vectors unwritten), is detected on the
 *              device and reported by kd_read_status().  No call traps or aborts.
 *  Supported n: 1 <= n <= 16384 whose prime factors all lie in
 *              {2, 3, 5, 7, 11, 13, 43} (kd_supported()).  Sixteen lengths have a
 *              compiled, tuned plan (kd_tuned()): 16, 32, 64, 128, 256, 512, 768,
 *              1024, 1536, 2048, 3072, 4096, 8192, 11008, 14336, 16384.  Every other
 *              supported length runs a run-time-length path (transform radices
 *              chosen per call, the pair held in shared memory): same method and
 *              outputs, several times slower.  Code words per vector: ceil(n/16),
 *              the last one padded with zero codes.
 */
#ifndef KASHIN_H
#define KASHIN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  KD_OK = 0,
  KD_ERR_INVALID_ARG = 1,   /* null required pointer, bad size, bad enum, ld too small */
  KD_ERR_UNSUPPORTED_N = 2, /* vector length outside the supported set (see "Supported n") */
  KD_ERR_CUDA = 3,          /* a CUDA runtime call or launch failed */
  KD_ERR_NONFINITE = 4,     /* a decomposed vector held NaN or Inf (device-detected) */
  KD_ERR_WORKSPACE = 5,     /* workspace pointer null, not 16-byte aligned, or too small */
  KD_ERR_TIMEOUT = 6        /* a bounded wait inside a kernel expired (device-detected) */
} kd_status;

typedef enum { KD_F32 = 0, KD_F16 = 1, KD_BF16 = 2 } kd_dtype;

typedef enum { KD_VEC_ROWS = 0, KD_VEC_COLUMNS = 1 } kd_layout;

/* Human-readable name of a status code (static string, never NULL). */
const char* kd_status_string(kd_status s);

/* Library version string. */
const char* kd_version(void);

/* KD_OK if vector length n is supported (see "Supported n" above), else
 * KD_ERR_UNSUPPORTED_N. */
kd_status kd_supported(int64_t n);

/* 1 if vector length n has a compiled, tuned plan, else 0 (unsupported lengths
 * included).  Informational: every supported n runs through the same calls. */
int kd_tuned(int64_t n);

/* Bytes of device workspace kd_decompose / kd_apply_p / kd_reconstruct need for
 * vector length n on the current device (0 if n is unsupported).  The workspace
 * holds the per-call sign mask, the transform twiddles and a device status word;
 * it must stay allocated until the enqueued work completes and must not be
 * shared by calls in flight on different streams. */
size_t kd_workspace_size(int64_t n);

/* The sign set eps of Sec. 3.1 / App. C for a seed, on the host:
 * eps_host[j] = +1 or -1, j < n.  Pure host computation, no CUDA call. */
kd_status kd_signs(uint64_t sign_seed, int64_t n, int8_t* eps_host);

/* Algorithm 1 on every vector of w, then the closed-form 2-bit coding of both
 * factors (Sec. 3.2 Algorithm 1; Sec. 2.1; App. C storage format).
 *
 *  w          input, dtype elements, `layout` with leading dimension ld.
 *  iters      k blocks (0 <= k <= 65536) of four atomic greedy steps (two on Q_N -> u,
 *             two on P Q_N -> vhat).  k = 0 gives zero factors, zero centres, codes 0.
 *  kmeans_iters  0..64 Lloyd refinement iterations of each factor's 4 centres from
 *             the closed form (Sec. 2.1 refines the closed-form centres with a few
 *             k-means iterations): every entry goes to its nearest centre (ties to the
 *             lower), each centre becomes its cluster's mean, an empty cluster keeps
 *             its centre.  0 = the closed-form centres alone.
 *  codes_u,   required, uint32[m][ceil(n/16)]: 2-bit code of u_i (resp. vhat_i) at
 *  codes_v    bits 2*(i%16) of word i/16 of vector j's row; code c indexes the
 *             ascending centre table.
 *  centres_u, required, float[m][4] ascending: -(a1+a2), -|a1-a2|, |a1-a2|, a1+a2
 *  centres_v  with (a1, a2) = (c1, c2) for u and (d1, d2) for vhat, or their
 *             refinement when kmeans_iters > 0.
 *  coeffs     optional, float[m][4]: c1, c2, d1, d2 (block-0 step coefficients).
 *  u, vhat,   optional, float[m][n] (vector-major, contiguous): the factors u_k,
 *  resid      vhat_k and the residual r_k of Algorithm 1, x = u + P vhat + r.
 *  trace      optional, int8[m][4*iters + 2*kmeans_iters][n]: rows 0..4k-1 hold the
 *             sign(.) in {-1, 0, +1} every atomic step applied to element i (natural
 *             order); rows 4k + 2t + f hold the cluster (0..3) of factor f (0 = u,
 *             1 = vhat) in refinement iteration t.  Test/debug output; enabling it
 *             does not change any other output bit.
 *  workspace  device scratch, 16-byte aligned (as cudaMalloc returns), of
 *             ws_bytes >= kd_workspace_size(n).
 *
 * Errors (returned before anything is enqueued): KD_ERR_INVALID_ARG for a bad size,
 * count or enum, ld too small, a null required pointer with m > 0, or a pointer not
 * aligned to its element (w to its dtype, codes and fp32 outputs to 4 bytes);
 * KD_ERR_UNSUPPORTED_N; KD_ERR_WORKSPACE.  KD_ERR_CUDA if a launch fails.
 *
 * Vectors are processed two at a time (2j, 2j+1); each vector's results depend
 * only on its own data and its pair partner's (through rounding only). */
kd_status kd_decompose(const void* w, kd_dtype dtype, kd_layout layout, int64_t n, int64_t m,
                       int64_t ld, uint64_t sign_seed, int iters, int kmeans_iters,
                       uint32_t* codes_u, uint32_t* codes_v, float* centres_u, float* centres_v,
                       float* coeffs, float* u, float* vhat, float* resid, int8_t* trace,
                       void* workspace, size_t ws_bytes, void* stream);

/* kd_decompose without a caller workspace, for callers that cannot allocate device
 * memory (a plugin whose host application owns every device allocation and forbids
 * direct cudaMalloc, or a loop that cannot afford cudaMalloc's implicit
 * synchronisation).  The paper has no counterpart: this is a library convenience.
 * Same arguments and results as kd_decompose minus workspace/ws_bytes; the scratch
 * lives in a 160 KB static device array inside the library instead.
 *   - Arguments are checked first, in kd_decompose's order and with its error codes;
 *     then n must be at most 8192 and its tables must fit the array (the tuned
 *     lengths; the run-time-length path needs per-CTA slots that do not fit),
 *     otherwise KD_ERR_WORKSPACE.  Nothing is enqueued on any error.
 *   - Allocates nothing.  Every GPU that loads the library holds the array until exit.
 *   - All calls share the array (it keeps the last call's tables); each call rewrites
 *     what it needs and clears the status word on its own stream, so calls that
 *     overlap on the GPU race.
 *   - The first call on a device resolves the array's address (cudaGetSymbolAddress,
 *     once per device): make that first call before any stream capture.
 *   - A non-finite input sets the status word in the array; kd_read_status_static
 *     reads it back. */
kd_status kd_decompose_static(const void* w, kd_dtype dtype, kd_layout layout, int64_t n, int64_t m,
                              int64_t ld, uint64_t sign_seed, int iters, int kmeans_iters,
                              uint32_t* codes_u, uint32_t* codes_v, float* centres_u, float* centres_v,
                              float* coeffs, float* u, float* vhat, float* resid, int8_t* trace,
                              void* stream);

/* kd_read_status for kd_decompose_static: synchronises `stream`, then returns
 * KD_ERR_TIMEOUT or KD_ERR_NONFINITE as kd_read_status does for the last
 * kd_decompose_static call on the current device, KD_OK otherwise (also when no
 * static call ran yet), and KD_ERR_CUDA if a CUDA call fails.  Allocates nothing.  The word is shared like the
 * rest of the array: a static call enqueued after the one of interest clears it. */
kd_status kd_read_status_static(void* stream);

/* ---------------------------------------------------------------------------
 * Several matrices of one vector length n in one launch (Algorithm 1 and the 2-bit
 * coding, as kd_decompose): the vector pairs of all matrices share the persistent
 * CTAs, so small matrices fill the GPU and the last wave of one matrix overlaps the
 * next.  Each matrix keeps its own sign seed, leading dimension and outputs; the
 * arithmetic per vector pair is identical to kd_decompose's (bitwise equal results).
 * Tuned lengths n <= 8192 run as one launch; longer vectors (which fill the GPU
 * alone) and the run-time-length path run one launch per matrix, in order, on the
 * same stream and workspace.
 *
 *   mats      HOST array of `count` descriptors (1 <= count <= KD_MAX_BATCH); read
 *             during the call only.  In each: w, m, ld, sign_seed as kd_decompose's
 *             arguments; codes_u, codes_v, centres_u, centres_v required (m > 0);
 *             coeffs optional (NULL).  No u / vhat / resid / trace outputs.
 *   dtype, layout, n, iters, kmeans_iters   shared by all matrices.
 *   workspace at least kd_workspace_size_batch(n, count) bytes.
 * Errors as kd_decompose. */
#define KD_MAX_BATCH 32
typedef struct kd_matrix {
  const void* w;
  int64_t m;
  int64_t ld;
  uint64_t sign_seed;
  uint32_t* codes_u;
  uint32_t* codes_v;
  float* centres_u;
  float* centres_v;
  float* coeffs;
} kd_matrix;

size_t kd_workspace_size_batch(int64_t n, int count);
kd_status kd_decompose_batch(const kd_matrix* mats, int count, kd_dtype dtype, kd_layout layout, int64_t n,
                             int iters, int kmeans_iters, void* workspace, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * kd_decompose_batch from HOST memory to HOST memory: the end-to-end call of a caller
 * that holds the weights on the host (Algorithm 1 and the 2-bit coding, as
 * kd_decompose_batch).  Every pointer in the descriptors is HOST memory; pinned memory
 * (cudaHostAlloc / cudaHostRegister) lets the copies run asynchronously, pageable
 * memory makes them synchronous.  On `stream`, in order: one host-to-device copy per
 * matrix input into `staging`, the batched decomposition, one device-to-host copy per
 * output.  The call returns once this is enqueued; the host outputs are valid after
 * the stream synchronises.  The host inputs must stay unchanged and the outputs
 * untouched until then.  Several calls may be in flight on different streams, each
 * with its own staging and workspace.
 *
 *   mats      HOST array of `count` descriptors (1 <= count <= KD_MAX_BATCH), read
 *             during the call: w as kd_decompose's input (m vectors, layout and ld; the
 *             whole m x ld block (KD_VEC_ROWS) or n x ld block (KD_VEC_COLUMNS) is
 *             copied), codes_u, codes_v (m x ceil(n/16) uint32), centres_u, centres_v
 *             (m x 4 fp32) required when m > 0, coeffs (m x 4) optional (NULL).
 *   staging   device memory, 256-byte aligned, at least kd_staging_size_host() bytes:
 *             the inputs and outputs on the device.  The library allocates nothing.
 *   workspace at least kd_workspace_size_batch(n, count) bytes, as kd_decompose_batch.
 * Errors: as kd_decompose_batch (argument checks first), KD_ERR_WORKSPACE for a null,
 * unaligned or short staging buffer, KD_ERR_CUDA if a copy or launch fails to enqueue.
 * The paper has no counterpart: this is the library's own end-to-end entry point. */
typedef struct kd_matrix_host {
  const void* w;
  int64_t m;
  int64_t ld;
  uint64_t sign_seed;
  uint32_t* codes_u;
  uint32_t* codes_v;
  float* centres_u;
  float* centres_v;
  float* coeffs;
} kd_matrix_host;

/* Device staging bytes kd_decompose_batch_host needs for these matrices (0 for an
 * invalid count, size or enum). */
size_t kd_staging_size_host(const kd_matrix_host* mats, int count, kd_dtype dtype, kd_layout layout, int64_t n);

kd_status kd_decompose_batch_host(const kd_matrix_host* mats, int count, kd_dtype dtype, kd_layout layout,
                                  int64_t n, int iters, int kmeans_iters, void* staging, size_t staging_bytes,
                                  void* workspace, size_t ws_bytes, void* stream);

/* y_j = P x_j for m vectors of length n, fp32, vector-major [m][n] contiguous
 * (Sec. 3.1: P z = IDCT(eps * DCT(z)); App. C uses the same operator on the rows
 * of the activations, XP).  x and y may alias; both 4-byte aligned
 * (KD_ERR_INVALID_ARG otherwise). */
kd_status kd_apply_p(const float* x, float* y, int64_t n, int64_t m, uint64_t sign_seed,
                     void* workspace, size_t ws_bytes, void* stream);

/* kd_apply_p for several matrices of one vector length n in one launch (the XP of a
 * layer's products, App. C), each with its own rows, output and sign seed:
 *   mats       HOST array of 1 <= count <= KD_MAX_BATCH descriptors, read during the call;
 *              y_j = P x_j for the m rows of x ([m][n] fp32 contiguous), x and y may alias.
 *   workspace  16-byte aligned, ws_bytes >= kd_workspace_size_batch(n, count).
 * Results equal kd_apply_p's per matrix, bit for bit.  Lengths above 8192 and the
 * run-time-length path run one launch per matrix, in order, on the same stream and
 * workspace.  Errors as kd_apply_p (the first invalid matrix's), and
 * KD_ERR_INVALID_ARG for a bad count or a null array. */
typedef struct kd_pmat {
  const float* x;
  float* y;
  int64_t m;
  uint64_t sign_seed;
} kd_pmat;

kd_status kd_apply_p_batch(const kd_pmat* mats, int count, int64_t n, void* workspace, size_t ws_bytes,
                           void* stream);

/* P's tables derived once, for serving: kd_prepare_p writes the twiddle table and the
 * sign sets of seeds[0..count) (set i from seeds[i]) into the workspace, on `stream`;
 * kd_apply_p_prepared then applies P to the rows of each matrix as kd_apply_p_batch does,
 * matrix i with sign set i, without deriving the tables again (its descriptors'
 * sign_seed fields are not read).  The two calls take the same n, count and workspace
 * (16-byte aligned, ws_bytes >= kd_workspace_size_batch(n, count)); results equal
 * kd_apply_p_batch's with the same seeds, bit for bit.  The tables stay valid until
 * another call writes that workspace.  Errors as kd_apply_p_batch (seeds null:
 * KD_ERR_INVALID_ARG). */
kd_status kd_prepare_p(const uint64_t* seeds, int count, int64_t n, void* workspace, size_t ws_bytes,
                       void* stream);
kd_status kd_apply_p_prepared(const kd_pmat* mats, int count, int64_t n, void* workspace, size_t ws_bytes,
                              void* stream);

/* Dense re-materialisation W_hat = U_q + P V_q (App. C): vector j of w_hat is
 * centres_u[j][code_u] + P(centres_v[j][code_v]).  Inputs as produced by
 * kd_decompose (centres 16-byte aligned, codes 4-byte aligned, KD_ERR_INVALID_ARG
 * otherwise); output dtype out_dtype in `layout` with leading dimension ld, aligned
 * to its element. */
kd_status kd_reconstruct(const uint32_t* codes_u, const uint32_t* codes_v,
                         const float* centres_u, const float* centres_v, int64_t n, int64_t m,
                         uint64_t sign_seed, kd_dtype out_dtype, kd_layout layout, void* w_hat,
                         int64_t ld, void* workspace, size_t ws_bytes, void* stream);

/* kd_reconstruct for several matrices of one vector length n in one launch (App. C
 * at load time: a layer's matrices together), each with its own codes, centres, sign
 * seed, output and ld; out_dtype and layout are shared.  Every matrix is written
 * exactly as kd_reconstruct would write it.
 *   mats       HOST array of `count` descriptors (1 <= count <= KD_MAX_BATCH), read
 *              during the call.
 *   workspace  16-byte aligned, ws_bytes >= kd_workspace_size_batch(n, count) (one
 *              sign set per matrix).
 * Lengths above 8192 run one launch per matrix, in order, on the same stream and
 * workspace.  Errors as kd_reconstruct (the first invalid matrix's), and
 * KD_ERR_INVALID_ARG for a bad count or a null array. */
typedef struct kd_recmat {
  const uint32_t* codes_u;
  const uint32_t* codes_v;
  const float* centres_u;
  const float* centres_v;
  uint64_t sign_seed;
  void* w_hat;
  int64_t m;
  int64_t ld;
} kd_recmat;

kd_status kd_reconstruct_batch(const kd_recmat* mats, int count, int64_t n, kd_dtype out_dtype, kd_layout layout,
                               void* workspace, size_t ws_bytes, void* stream);

/* Synchronises `stream` and reads the status word of the last kd_decompose (or
 * kd_decompose_batch) on this workspace: KD_ERR_TIMEOUT if a staged-input copy did
 * not complete within the kernel's bounded wait (about a second; that CTA's
 * remaining vectors are not written), else KD_ERR_NONFINITE if any vector held a
 * NaN or Inf, KD_OK otherwise (KD_ERR_CUDA if the synchronisation fails). */
kd_status kd_read_status(const void* workspace, void* stream);

/* Dequantise one 2-bit factor plane (App. C, inference): out entry i of vector j =
 * centres[j*4 + code_j(i)], code_j(i) = bits 2(i%16)..2(i%16)+1 of codes[j*ceil(n/16) + i/16].
 * With U_q and V_q expanded this way the layer product folds as
 *   X W = X U_q + (X P) V_q = [X | XP] [U_q; V_q]      (App. C, Eq. inference_factor),
 * XP from kd_apply_p on the rows of X; kd_reconstruct gives W_hat = U_q + P V_q itself.
 *   codes    device, m x ceil(n/16) uint32 (kd_decompose's codes_u or codes_v).
 *   centres  device, m x 4 fp32 ascending (centres_u or centres_v), 16-byte aligned.
 *   out      device, dtype out_dtype, layout as for kd_decompose's input (ld >= n for
 *            KD_VEC_ROWS, >= m for KD_VEC_COLUMNS).
 * No workspace.  Errors: KD_ERR_INVALID_ARG (sizes, enums, ld, null or unaligned
 * pointers with m > 0), KD_ERR_CUDA (launch).  m == 0 enqueues nothing. */
kd_status kd_dequantise(const uint32_t* codes, const float* centres, int64_t n, int64_t m, kd_dtype out_dtype,
                        kd_layout layout, void* out, int64_t ld, void* stream);

/* kd_dequantise for several planes of one vector length n in one launch (App. C at
 * load time: a layer's U_q and V_q planes together), so that small planes do not
 * each pay a launch and a partly filled last wave.
 *   planes  HOST array of `count` descriptors (1 <= count <= KD_MAX_BATCH), read
 *           during the call; each as kd_dequantise's codes, centres, m, out and ld.
 * Every plane is written exactly as kd_dequantise would write it; outputs that
 * overlap give undefined contents.  Errors as kd_dequantise (the first invalid
 * plane's), and KD_ERR_INVALID_ARG for a bad count or a null array. */
typedef struct kd_plane {
  const uint32_t* codes;
  const float* centres;
  void* out;
  int64_t m;
  int64_t ld;
} kd_plane;

kd_status kd_dequantise_batch(const kd_plane* planes, int count, int64_t n, kd_dtype out_dtype, kd_layout layout,
                              void* stream);

/* Measured FP32 throughput of the current device in TFLOP/s (packed FFMA2 chains on
 * every SM, best of three timed launches on `stream`; synchronises the stream).
 * Used as the measured denominator of the transform kernels' ALU roofline. */
kd_status kd_measure_fp32_peak(double* tflops, void* stream);

/* The layer product straight from the 2-bit planes (App. C: X W = X U_q + (X P) V_q =
 * [X | XP] [U_q; V_q], evaluated without expanding U_q or V_q):
 *   y[r*ldy + j] = sum_i centres_u[j][code_u(j,i)] x[r*ldx + i]
 *                + sum_i centres_v[j][code_v(j,i)] xp[r*ldx + i],   r < batch, j < m,
 * i.e. Y = X W_hat^T for the m vectors (output channels) of W_hat = U_q + P V_q.
 *   codes_u, codes_v   device, m x ceil(n/16) uint32, 4-byte aligned (kd_decompose's).
 *   centres_u, _v      device, m x 4 fp32 ascending, 16-byte aligned.
 *   x                  device fp32, batch rows of n inputs, row r at x + r*ldx (ldx >= n).
 *   xp                 device fp32, the same rows times P (kd_apply_p with the matrix's
 *                      sign seed on the rows of X), same layout and ldx.
 *   y                  device fp32, batch rows of m outputs, row r at y + r*ldy (ldy >= m).
 * Every code word is read once per group of up to two batch rows; accumulation is
 * fp32 in a fixed order (deterministic).  Errors: KD_ERR_INVALID_ARG (sizes, null or
 * unaligned pointers when m > 0 and batch > 0), KD_ERR_CUDA (launch).  m == 0 or
 * batch == 0 enqueues nothing. */
kd_status kd_matmul_2bit(const uint32_t* codes_u, const uint32_t* codes_v, const float* centres_u,
                         const float* centres_v, int64_t n, int64_t m, const float* x, const float* xp,
                         int64_t batch, int64_t ldx, float* y, int64_t ldy, void* stream);

/* kd_matmul_2bit for several matrices in one launch (a layer's products for one batch
 * of activations): each descriptor as kd_matmul_2bit's arguments, each matrix with its
 * own n, m, inputs and output.  mats is a HOST array of 1 <= count <= KD_MAX_BATCH
 * descriptors read during the call.  Results equal kd_matmul_2bit's per matrix, bit for
 * bit.  Errors as kd_matmul_2bit (the first invalid matrix's), and KD_ERR_INVALID_ARG
 * for a bad count or a null array. */
typedef struct kd_fold_mat {
  const uint32_t* codes_u;
  const uint32_t* codes_v;
  const float* centres_u;
  const float* centres_v;
  const float* x;
  const float* xp;
  float* y;
  int64_t n;
  int64_t m;
  int64_t ldx;
  int64_t ldy;
} kd_fold_mat;

kd_status kd_matmul_2bit_batch(const kd_fold_mat* mats, int count, int64_t batch, void* stream);

/* The layer product of kd_matmul_2bit for fp16 activations, on the tensor cores:
 *   y[r*ldy + j] = sum_i h(centres_u[j][code_u(j,i)]) x[r*ldx + i]
 *                + sum_i h(centres_v[j][code_v(j,i)]) xp[r*ldx + i],   r < batch, j < m,
 * where x and xp are fp16 (IEEE binary16) and h() rounds a centre to fp16 (nearest,
 * ties to even); products are exact and the sums are fp32 (mma.sync m16n8k16).  This
 * is Y = X W_hat^T in the precision of a dense fp16 layer: the activations and the
 * weights' values are fp16, nothing else is rounded.
 *   codes_u, codes_v, centres_u, centres_v, n, m, batch, y, ldy as in kd_matmul_2bit.
 *   x, xp   device fp16, batch rows of n inputs, row r at x + r*ldx (ldx >= n);
 *           xp holds the rows of X P (kd_apply_p, rounded to fp16 by the caller).
 *           2-byte aligned; 16-byte aligned rows (base and ldx a multiple of 8) take
 *           128-bit loads.
 * The centres must be finite in fp16 (|c| <= 65504): a code padding past n multiplies
 * a zero input by a centre.  Every code word is read once per group of up to 16 batch
 * rows; the sums run in a fixed order (deterministic).  Errors and empty calls as
 * kd_matmul_2bit. */
kd_status kd_matmul_2bit_f16(const uint32_t* codes_u, const uint32_t* codes_v, const float* centres_u,
                             const float* centres_v, int64_t n, int64_t m, const void* x, const void* xp,
                             int64_t batch, int64_t ldx, float* y, int64_t ldy, void* stream);

/* kd_matmul_2bit_f16 for several matrices in one launch per 16 batch rows; each
 * descriptor as kd_matmul_2bit_f16's arguments.  mats is a HOST array of 1 <= count <=
 * KD_MAX_BATCH descriptors.  Results equal kd_matmul_2bit_f16's per matrix, bit for bit.
 * Errors as kd_matmul_2bit_batch. */
typedef struct kd_fold_mat_f16 {
  const uint32_t* codes_u;
  const uint32_t* codes_v;
  const float* centres_u;
  const float* centres_v;
  const void* x;
  const void* xp;
  float* y;
  int64_t n;
  int64_t m;
  int64_t ldx;
  int64_t ldy;
} kd_fold_mat_f16;

kd_status kd_matmul_2bit_f16_batch(const kd_fold_mat_f16* mats, int count, int64_t batch, void* stream);

/* kd_matmul_2bit_f16 and its batched form for bf16 activations: x and xp are bf16, each
 * centre is rounded to bf16 (nearest, ties to even), products are exact and sums fp32
 * (mma.sync m16n8k16 .bf16).  Arguments, layouts, alignment and errors as the fp16
 * calls (the descriptor struct is shared). */
kd_status kd_matmul_2bit_bf16(const uint32_t* codes_u, const uint32_t* codes_v, const float* centres_u,
                              const float* centres_v, int64_t n, int64_t m, const void* x, const void* xp,
                              int64_t batch, int64_t ldx, float* y, int64_t ldy, void* stream);
kd_status kd_matmul_2bit_bf16_batch(const kd_fold_mat_f16* mats, int count, int64_t batch, void* stream);

/* ---------------------------------------------------------------------------
 * Randomized-Hadamard incoherence rotation (Sec. 4, the "+H" of Kashin-DCT+H:
 * the weights are rotated by a randomized Hadamard transform before the
 * decomposition).  The paper does not give the construction; this library's:
 *
 *   forward   y_j = (I_{n/b} (x) H_b / sqrt(b)) diag(s) x_j
 *   inverse   y_j = diag(s) (I_{n/b} (x) H_b / sqrt(b)) x_j       (the transpose)
 *
 * for every vector j, with H_b the Sylvester Hadamard matrix (H_1 = [1],
 * H_2k = [[H_k, H_k], [H_k, -H_k]]) applied to each contiguous block of b
 * entries, b = kd_rht_block(n) (the largest power of two dividing n, at most
 * 16384), and s_i = -1 where bit 63 of SplitMix64(seed + (i+1)*0x9E3779B97F4A7C15)
 * is set, +1 otherwise (the same generator as the decomposition's eps; give the
 * rotation its own seed).
 *
 *   x        device, m vectors of n entries, vector j at x[j*ldx + i] (ldx >= n),
 *            dtype KD_F32 / KD_F16 / KD_BF16.
 *   y        device fp32, vector j at y[j*ldy + i] (ldy >= n).  y may be x itself
 *            (in place) when dtype is KD_F32 and ldy == ldx; other overlaps are
 *            the caller's error.
 *   inverse  0 = forward, 1 = inverse.
 *   status   optional device word (NULL = none).  The kernel streams its input
 *            through shared memory with bulk copies and bounds every wait for
 *            one; if a copy has not landed after about a second it ORs
 *            KD_RHT_ERR_TIMEOUT into *status, leaves that part of y unwritten
 *            and returns.  The caller clears the word and reads it back.
 *   stream   cudaStream_t as void*.
 * Errors: KD_ERR_UNSUPPORTED_N unless n % 16 == 0 and 16 <= n <= 65536;
 * KD_ERR_INVALID_ARG for m < 0, ld too small, bad dtype or flag, null pointers
 * with m > 0, x, y or status not aligned to their elements, or an in-place call
 * that is not fp32 with equal strides;
 * KD_ERR_CUDA if the launch fails.  m == 0 enqueues nothing.  No workspace.
 * To rotate along the other axis of a matrix (the output side of a two-sided
 * rotation) pass its transpose. */
#define KD_RHT_ERR_TIMEOUT 1u
int64_t kd_rht_block(int64_t n); /* block length b for vectors of length n, 0 if unsupported */
kd_status kd_rht(const void* x, kd_dtype dtype, int64_t n, int64_t m, int64_t ldx, uint64_t seed, int inverse,
                 float* y, int64_t ldy, uint32_t* status, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* KASHIN_H */
