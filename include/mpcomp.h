/*
 * mpcomp.h -- C ABI of libmpcomp, GB300 (sm_103a) kernels for the activation and
 * gradient compression operators of Rudakov, Beznosikov, Kholodov and Gasnikov,
 * "Activations and Gradients Compression for Model-Parallel Training"
 * (arXiv 2401.07788).
 *
 * The operators compress a tensor that crosses a model-parallel stage boundary:
 * activations in the forward pass, their gradients in the backward pass (§2.1).
 *
 * Conventions for every entry point
 * ---------------------------------
 *  - Tensors are row-major fp32 matrices [rows][row_len]; each operator acts on
 *    every row independently (the vector the paper compresses, §2.2, §2.3).
 *  - Every pointer argument is CUDA device memory owned by the caller, except
 *    where a comment says otherwise.  The library allocates no device memory.
 *  - Every call is asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *    default stream).  Arguments are validated on the host before any launch;
 *    an invalid call returns an error code and launches nothing.
 *  - Inputs must not alias outputs or state buffers, except where noted.
 *  - Inputs are assumed finite.  Non-finite values give defined but unspecified
 *    outputs; they never cause out-of-bounds accesses.
 *  - Errors found on the device (an out-of-range sample id, a timed-out wait)
 *    are recorded in a per-process device status word and reported by
 *    mpc_get_status(); the outputs of the failing call are then unspecified.
 *  - No C++ exception crosses this interface.
 *  - The library looks up per-device addresses of its device variables once
 *    per device and keeps them: it supports the device's primary context only
 *    (the CUDA runtime's), and no cudaDeviceReset while it is loaded.
 *
 * TopK payload: for each row, the k kept entries as `vals[rows][k]` (fp32, the
 * exact bits of the kept value, sign included) and `idx[rows][k]` (int32 column
 * within the row), listed by ascending column.  The kept set is the k entries
 * of largest magnitude; entries of equal magnitude are taken lower column
 * first, so the result is unique.
 *
 * Quantisation payload: `codes[rows][W]` uint32 words, W from
 * mpc_quant_codes_words()/rows, holding the row's codes as an LSB-first
 * bitstream (code j in bits [j*bits, j*bits+bits); bit p in word p/32, bit
 * p%32), zero-padded so that each row starts on a 16-byte boundary; plus
 * `scale[rows]` and `minv[rows]` (fp32).
 */
#ifndef MPCOMP_H
#define MPCOMP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Layout-compatible with cudaStream_t. */
typedef struct CUstream_st* mpc_stream_t;

typedef enum {
    MPC_OK = 0,
    MPC_ERR_INVALID_ARG = 1, /* bad size, null or misaligned pointer, bad enum */
    MPC_ERR_UNSUPPORTED = 2, /* valid request the library does not implement */
    MPC_ERR_WORKSPACE = 3,   /* workspace missing or smaller than required */
    MPC_ERR_CUDA = 4,        /* a CUDA runtime call or launch failed */
    MPC_ERR_TIMEOUT = 5,     /* a device-side wait gave up (see mpc_get_status) */
    MPC_ERR_DEVICE = 6       /* a device-side check failed (see mpc_get_status) */
} mpc_status;

typedef enum {
    MPC_ROUND_NEAREST = 0,   /* round half to even */
    MPC_ROUND_STOCHASTIC = 1 /* floor(t + u), u from the counter-based generator */
} mpc_rounding;

/* Library version as 10000*major + 100*minor + patch. */
int mpc_version(void);

/* ------------------------------------------------------------------------ */
/* TopK sparsification (§2.3)                                               */
/* ------------------------------------------------------------------------ */

/* Bytes of device workspace the TopK compress calls below need for this
 * shape (0 when none).  Rows longer than the on-chip path handles (65536
 * entries) use a multi-pass path that keeps counters, lists and candidates
 * in the workspace; it takes the rows in batches of up to 64 (about 2^26
 * entries a batch), one 256-byte-aligned slice of the workspace per row of a
 * batch, so the size grows with min(rows, batch) rather than with rows. */
size_t mpc_topk_workspace_bytes(int64_t rows, int64_t row_len, int64_t k);

/* TopK compress (§2.3: keep the K% entries of each row with the largest
 * magnitudes).
 *   x     [rows][row_len] fp32, read only.
 *   k     entries kept per row, 1 <= k <= row_len (the caller turns K% into k).
 *   vals  [rows][k] fp32, out;  idx [rows][k] int32, out (ascending per row).
 *   ws    workspace of ws_bytes >= mpc_topk_workspace_bytes(rows, row_len, k)
 *         (may be NULL when that is 0).
 * Requires 1 <= row_len <= 2^31-1, rows >= 0 (0 is a no-op). */
mpc_status mpc_topk_compress(const float* x, int64_t rows, int64_t row_len, int64_t k,
                             float* vals, int32_t* idx, void* ws, size_t ws_bytes,
                             mpc_stream_t stream);

/* TopK decompress (§2.3: the kept values back at their columns, zero
 * elsewhere):
 *   y [rows][row_len] = +0 everywhere except y[r][idx[r][i]] = vals[r][i].
 * idx must be strictly ascending in each row and within [0, row_len) (as
 * produced by the compress calls); entries that are not are skipped, never
 * written out of bounds. */
mpc_status mpc_topk_decompress(const float* vals, const int32_t* idx, int64_t rows,
                               int64_t row_len, int64_t k, float* y,
                               mpc_stream_t stream);

/* TopK index reuse (§3.2, Table 5: the gradient at a boundary is compressed
 * at the TopK indices of the activation, which fine-tuning needs to converge):
 *   vals[r][i] = g[r][idx[r][i]]  (bit copy), for 0 <= i < k.
 *   g     [rows][row_len] fp32, read only (device memory).
 *   idx   [rows][k] int32, read only: the payload indices of a compress call
 *         on the tensor g pairs with (any order is accepted).
 *   vals  [rows][k] fp32, out; decompress with mpc_topk_decompress(vals, idx).
 * An index outside [0, row_len) reads nothing: its value is +0 and
 * mpc_get_status then reports MPC_ERR_DEVICE.  Requires 1 <= k <= row_len. */
mpc_status mpc_topk_gather(const float* g, int64_t rows, int64_t row_len, const int32_t* idx,
                           int64_t k, float* vals, mpc_stream_t stream);

/* Error feedback of Seide et al. fused with TopK (§2.4: the message is
 * C(X + e) and the error kept is e = X - C(X), one global buffer per
 * operator carried across batches):
 *   s = x + err (fp32, round to nearest);  (vals, idx) = TopK(s, k);
 *   err <- s - C(s), i.e. +0 at the kept entries and s elsewhere.
 * err [rows][row_len] is read and rewritten in place (start it at zero). */
mpc_status mpc_ef_topk_compress(const float* x, float* err, int64_t rows, int64_t row_len,
                                int64_t k, float* vals, int32_t* idx, void* ws,
                                size_t ws_bytes, mpc_stream_t stream);

/* EF-mixed TopK (§2.4: half of the K% budget goes to the largest entries of
 * the input and half to the largest of the error buffer; input and buffer are
 * summed and sent on those K% positions).  Reading: the
 * input's share is its ceil(k/2) largest |x|; the buffer's share is its
 * floor(k/2) largest |err| among the entries the input's share did not take
 * (so exactly k entries are sent); ties go to the lower index.  Then
 *   s = x + err;  (vals, idx) = s at those k entries, ascending idx;
 *   err <- +0 there and s elsewhere.
 * err [rows][row_len] is read and rewritten in place (start it at zero).
 * ws: device workspace of ws_bytes >= mpc_efmix_workspace_bytes(rows,
 * row_len, k), 256-byte aligned (never NULL: the input's share is kept there
 * between the two selections); MPC_ERR_WORKSPACE if smaller. */
size_t mpc_efmix_workspace_bytes(int64_t rows, int64_t row_len, int64_t k);
mpc_status mpc_efmix_topk_compress(const float* x, float* err, int64_t rows, int64_t row_len,
                                   int64_t k, float* vals, int32_t* idx, void* ws,
                                   size_t ws_bytes, mpc_stream_t stream);

/* EF21 fused with TopK (§2.4: message C(X_{i+1} - g_i), buffer
 * g_{i+1} = g_i + C(X_{i+1} - g_i)):
 *   d = x - g;  (vals, idx) = TopK(d, k);  g[kept] <- g[kept] + d[kept].
 * Entries of g off the support are left untouched (bit for bit).
 * g [rows][row_len] is updated in place (start it at zero). */
mpc_status mpc_ef21_topk_compress(const float* x, float* g, int64_t rows, int64_t row_len,
                                  int64_t k, float* vals, int32_t* idx, void* ws,
                                  size_t ws_bytes, mpc_stream_t stream);

/* ------------------------------------------------------------------------ */
/* AQ-SGD with TopK (§2.5)                                                  */
/* ------------------------------------------------------------------------ */

/* AQ-SGD sender (§2.5: the change of the activation against a buffer kept
 * per training sample is compressed and sent, and the buffer takes it):
 *   for i < n_ids, r < rows_per_sample, with s = sample_ids[i]:
 *     d = x[i][r] - buf[s][r];  payload row i*rows_per_sample + r = TopK(d, k);
 *     buf[s][r][kept] <- buf[s][r][kept] + d[kept].
 *   x          [n_ids][rows_per_sample][row_len] fp32.
 *   buf        [num_samples][rows_per_sample][row_len] fp32, in place
 *              (64-bit offsets; may exceed 2^31 elements).
 *   sample_ids device int64[n_ids], each in [0, num_samples), no duplicates
 *              (duplicates race; an id out of range sets MPC_ERR_DEVICE and
 *              its rows are skipped).
 *   vals, idx  [n_ids*rows_per_sample][k]. */
mpc_status mpc_aqsgd_compress(const float* x, float* buf, int64_t num_samples,
                              const int64_t* sample_ids, int64_t n_ids,
                              int64_t rows_per_sample, int64_t row_len, int64_t k,
                              float* vals, int32_t* idx, void* ws, size_t ws_bytes,
                              mpc_stream_t stream);

/* AQ-SGD receiver: its own copy of the per-sample buffer takes the same
 * update, buf_recv[s][r][idx] <- buf_recv[s][r][idx] + vals (the same fp32
 * addition as the sender's, so both copies stay bit-identical).  Same
 * shapes and id rules as mpc_aqsgd_compress. */
mpc_status mpc_aqsgd_decompress(const float* vals, const int32_t* idx, float* buf_recv,
                                int64_t num_samples, const int64_t* sample_ids,
                                int64_t n_ids, int64_t rows_per_sample, int64_t row_len,
                                int64_t k, mpc_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Min-max quantisation (§2.2)                                              */
/* ------------------------------------------------------------------------ */

/* Total uint32 words of `codes` for this shape: rows * W with
 * W = roundup4(ceil(row_len * bits / 32)).  bits in 1..16 (§2.2 evaluates 2,
 * 4, 6 and 8 bits; widths that do not divide 32, such as 6, have codes that
 * straddle two words) or 32; 0 for an unsupported width. */
size_t mpc_quant_codes_words(int64_t rows, int64_t row_len, int bits);

/* Bytes of device workspace mpc_quant_compress needs (0 for rows that the
 * single-pass kernel handles). */
size_t mpc_quant_workspace_bytes(int64_t rows, int64_t row_len, int bits);

/* Quantise (§2.2: each row scaled to [0, 1] by its minimum and maximum, then
 * rounded to one of 2^bits levels), per row, with L = 2^bits - 1:
 *   mn, mx = row minimum and maximum (-0 ordered below +0);
 *   scale = (mx - mn) / L;  inv = L / (mx - mn);  t = (x - mn) * inv;
 *   q = clamp(round_half_even(t), 0, L)            (MPC_ROUND_NEAREST) or
 *   q = clamp(floor(t + u), 0, L)                  (MPC_ROUND_STOCHASTIC),
 * every step one fp32 round-to-nearest operation.  A row whose range is 0
 * or whose range or inv is infinite sends codes 0, scale 0, minv = mn.
 * u for flat element i = row*row_len + j is (h >> 8) * 2^-24, where h is
 * the low (even i) or high (odd i) 32 bits of splitmix64 at counter i >> 1:
 * z = seed + (c+1)*0x9E3779B97F4A7C15, then the splitmix64 finaliser
 * (Steele, Lea & Flood, OOPSLA 2014).  The generator is not in the paper.
 * bits = 32 is a passthrough: codes hold the raw fp32 bits, scale = minv = 0.
 *   x      [rows][row_len] fp32.
 *   codes  mpc_quant_codes_words(rows, row_len, bits) uint32, out.
 *   scale, minv  [rows] fp32, out.  */
mpc_status mpc_quant_compress(const float* x, int64_t rows, int64_t row_len, int bits,
                              mpc_rounding mode, uint64_t seed, uint32_t* codes,
                              float* scale, float* minv, void* ws, size_t ws_bytes,
                              mpc_stream_t stream);

/* Dequantise (§2.2: the codes mapped back to the row's original range):
 * y = minv + float(q) * scale, two fp32 round-to-nearest operations
 * (bits = 32: y = the raw bits). */
mpc_status mpc_quant_decompress(const uint32_t* codes, const float* scale,
                                const float* minv, int64_t rows, int64_t row_len, int bits,
                                float* y, mpc_stream_t stream);

/* AQ-SGD with quantisation (§2.5: the change of each training sample's
 * activation against a buffer kept per sample is what travels; the cited work
 * compresses that change with the quantiser of §2.2):
 *   for i < n_ids, r < rows_per_sample, with s = sample_ids[i] and logical row
 *   l = i*rows_per_sample + r:
 *     d = x[i][r] - buf[s][r];  codes/scale/minv row l = Quant(d) exactly as
 *     mpc_quant_compress on the [n_ids*rows_per_sample][row_len] rows of d
 *     (the same seed gives the same stochastic draws);
 *     buf[s][r] <- buf[s][r] + Dequant(row l)   (fp32 round to nearest).
 *   x          [n_ids][rows_per_sample][row_len] fp32.
 *   buf        [num_samples][rows_per_sample][row_len] fp32, in place.
 *   sample_ids device int64[n_ids], each in [0, num_samples), no duplicates
 *              (duplicates race; an id out of range sets MPC_ERR_DEVICE, its
 *              d rows are taken as zero and its buffer rows are left alone).
 *   bits, mode as mpc_quant_compress; codes, scale, minv out as there.
 *   ws         device workspace of mpc_aqsgd_quant_workspace_bytes() bytes,
 *              8-byte aligned (always needed: it holds d).
 * One launch for 2/4/8-bit codes on rows of up to 4096 entries (d formed,
 * quantised and the buffer updated in the same pass; the workspace is then
 * unused); otherwise three (d, the quantiser, the buffer update),
 * stream-ordered. */
size_t mpc_aqsgd_quant_workspace_bytes(int64_t n_ids, int64_t rows_per_sample,
                                       int64_t row_len, int bits);
mpc_status mpc_aqsgd_quant_compress(const float* x, float* buf, int64_t num_samples,
                                    const int64_t* sample_ids, int64_t n_ids,
                                    int64_t rows_per_sample, int64_t row_len, int bits,
                                    mpc_rounding mode, uint64_t seed, uint32_t* codes,
                                    float* scale, float* minv, void* ws, size_t ws_bytes,
                                    mpc_stream_t stream);

/* AQ-SGD with quantisation, the receiver: its copy of the buffer takes the
 * same update, buf_recv[s][r] <- buf_recv[s][r] + Dequant(row l), with the
 * sender's fp32 operations, so the two copies stay bit-identical.  Shapes and
 * id rules as mpc_aqsgd_quant_compress. */
mpc_status mpc_aqsgd_quant_decompress(const uint32_t* codes, const float* scale,
                                      const float* minv, float* buf_recv, int64_t num_samples,
                                      const int64_t* sample_ids, int64_t n_ids,
                                      int64_t rows_per_sample, int64_t row_len, int bits,
                                      mpc_stream_t stream);

/* Quantise without allocating (the paper has no counterpart; this is a
 * deployment convenience).  Same operation, arguments and results as
 * mpc_quant_compress, bit for bit, but with no workspace argument: for callers
 * that cannot allocate device memory when they quantise (a fixed memory plan,
 * a host framework that forbids allocation inside its step, an allocator that
 * cannot be called from there).  The per-row scratch is a static device array
 * of 8 * MPC_QUANT_NOALLOC_MAX_ROWS bytes (512 KiB) that every device loading
 * the library keeps until the process exits.  rows > MPC_QUANT_NOALLOC_MAX_ROWS
 * returns MPC_ERR_INVALID_ARG and launches nothing.
 * Only calls whose rows are longer than 65536 entries (the two-pass path)
 * use the array; shorter rows run exactly as in mpc_quant_compress.
 * The first call on a device looks up the array's device address (with that
 * device current); make that first call outside any CUDA stream capture.
 * Every call with rows longer than 65536 entries shares the one array: such
 * calls whose kernels may overlap on the GPU (different streams without
 * ordering) race and give undefined results; calls ordered on one stream are
 * safe.  No cudaMalloc, cudaFree or allocating library routine is called. */
#define MPC_QUANT_NOALLOC_MAX_ROWS 65536
mpc_status mpc_quant_compress_noalloc(const float* x, int64_t rows, int64_t row_len, int bits,
                                      mpc_rounding mode, uint64_t seed, uint32_t* codes,
                                      float* scale, float* minv, mpc_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Status and diagnostics                                                   */
/* ------------------------------------------------------------------------ */

/* Synchronise `stream`, then read and clear the device status word that the
 * kernels set: MPC_ERR_TIMEOUT if a bounded wait gave up, MPC_ERR_DEVICE if a
 * device-side argument check failed, MPC_ERR_CUDA if the stream reported an
 * error, else MPC_OK. */
mpc_status mpc_get_status(mpc_stream_t stream);

/* Message describing the last error returned on the calling host thread
 * (empty string if none).  The pointer stays valid until the next call on
 * that thread. */
const char* mpc_last_error(void);

/* Test knobs (values persist for the process; not for production use):
 *   MPC_KNOB_SPIN_LIMIT   tries of a device-side wait before it gives up; the
 *                         wait also stops after about 64 ns x this value
 *                         (default 1<<20, about 0.07 s; 0 makes every first wait give
 *                         up, which tests the timeout report without a fault);
 *   MPC_KNOB_TOPK_PATH    0 = automatic, 1 = force the on-chip row path when
 *                         it fits, 2 = force the multi-pass (workspace) path,
 *                         3 = automatic but rows of 8193..65536 entries always
 *                         split over a cluster of CTAs (never one wide CTA nor
 *                         the two-pass row kernel),
 *                         4 = automatic but rows of 1025..65536 entries take
 *                         the cluster / CTA kernels instead of the band and
 *                         two-pass row kernels;
 *   MPC_KNOB_PDL          1 (default) = launch the hot kernels with
 *                         programmatic dependent launch, so that a launch
 *                         overlaps the end of the previous one in the stream
 *                         (every kernel first waits for the grids it depends
 *                         on); 0 = plain stream order.
 * Returns MPC_ERR_INVALID_ARG for an unknown knob or value. */
typedef enum { MPC_KNOB_SPIN_LIMIT = 1, MPC_KNOB_TOPK_PATH = 2, MPC_KNOB_PDL = 3 } mpc_knob;
mpc_status mpc_set_knob(mpc_knob knob, int64_t value);

#ifdef __cplusplus
}
#endif
#endif /* MPCOMP_H */
