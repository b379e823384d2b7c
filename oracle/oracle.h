/*
 * oracle.h -- declarations of the CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY.  The oracle is a plain, slow, single-threaded
 * restatement of the compression operators of Rudakov, Beznosikov, Kholodov
 * and Gasnikov, "Activations and Gradients Compression for Model-Parallel
 * Training" (arXiv 2401.07788).  It exists to check the CUDA library.  Only
 * tests/, __graft_entry__.smoke() and the CPU-baseline leg of bench.py may
 * load it.  It shares no code, header, table or helper with the CUDA path.
 *
 * Precision: the paper trains in fp32 (§3.1, §3.2); every operator below is a
 * fixed sequence of IEEE-754 binary32 round-to-nearest-even operations, built
 * with -ffp-contract=off so that no multiply-add is fused.
 *
 * Layout conventions (all row-major, caller-owned host memory):
 *   x, e, g, y     float[rows][row_len]
 *   vals, idx      float[rows][k], int32[rows][k]  (kept entries, ascending idx)
 *   buf            float[num_samples][rows_per_sample][row_len]
 *   codes          uint32[rows][W], W = orc_quant_row_words(row_len, bits)
 *   scale, minv    float[rows]
 */
#ifndef MPC_ORACLE_H
#define MPC_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* splitmix64 (Steele, Lea & Flood, OOPSLA 2014) evaluated at one counter:
 * the finaliser applied to seed + (counter + 1) * 0x9E3779B97F4A7C15. */
uint64_t orc_splitmix64(uint64_t seed, uint64_t counter);

/* Uniform u in [0, 1) for flat element index i: 24 bits of one 32-bit half
 * of splitmix64(seed, i >> 1) (low half for even i, high half for odd i). */
float orc_uniform(uint64_t seed, uint64_t i);

/* TopK, §2.3: keep the k entries of largest magnitude per row. */
void orc_topk_compress(const float* x, int64_t rows, int64_t row_len, int64_t k,
                       float* vals, int32_t* idx);
void orc_topk_decompress(const float* vals, const int32_t* idx, int64_t rows,
                         int64_t row_len, int64_t k, float* y);

/* TopK index reuse, §3.2 (Table 5): vals[r][i] = g[r][idx[r][i]]. */
void orc_topk_gather(const float* g, int64_t rows, int64_t row_len, const int32_t* idx,
                     int64_t k, float* vals);

/* Error feedback (Seide), §2.4: s = x + e, send C(s), e <- s - C(s). */
void orc_ef_topk_compress(const float* x, float* e, int64_t rows, int64_t row_len,
                          int64_t k, float* vals, int32_t* idx);

/* EF-mixed, §2.4: ceil(k/2) largest |x|, then floor(k/2) largest |e| among the
 * other entries; x + e sent there, e <- x + e elsewhere and +0 there. */
void orc_efmix_topk_compress(const float* x, float* e, int64_t rows, int64_t row_len,
                             int64_t k, float* vals, int32_t* idx);

/* EF21, §2.4: send C(x - g), g <- g + C(x - g). */
void orc_ef21_topk_compress(const float* x, float* g, int64_t rows, int64_t row_len,
                            int64_t k, float* vals, int32_t* idx);

/* AQ-SGD with TopK, §2.5: per-sample buffer; EF21 applied to buf[sample_ids[i]]. */
void orc_aqsgd_compress(const float* x, float* buf, int64_t num_samples,
                        const int64_t* sample_ids, int64_t n_ids,
                        int64_t rows_per_sample, int64_t row_len, int64_t k,
                        float* vals, int32_t* idx);
void orc_aqsgd_decompress(const float* vals, const int32_t* idx, float* buf_recv,
                          int64_t num_samples, const int64_t* sample_ids,
                          int64_t n_ids, int64_t rows_per_sample, int64_t row_len,
                          int64_t k);

/* Min-max quantisation, §2.2.  bits in 1..16 or 32 (32 = raw passthrough).
 * mode 0 = round to nearest (ties to even), 1 = stochastic rounding. */
int64_t orc_quant_row_words(int64_t row_len, int bits);
void orc_quant_compress(const float* x, int64_t rows, int64_t row_len, int bits,
                        int mode, uint64_t seed, uint32_t* codes, float* scale,
                        float* minv);
void orc_quant_decompress(const uint32_t* codes, const float* scale, const float* minv,
                          int64_t rows, int64_t row_len, int bits, float* y);

/* AQ-SGD with quantisation, §2.5: d = x - buf[id, r]; message Quant(d);
 * buf[id, r] <- buf[id, r] + Dequant(Quant(d)).  Codes as orc_quant_compress
 * on the gathered rows (logical row i * rows_per_sample + r). */
void orc_aqsgd_quant_compress(const float* x, float* buf, int64_t num_samples,
                              const int64_t* sample_ids, int64_t n_ids,
                              int64_t rows_per_sample, int64_t row_len, int bits, int mode,
                              uint64_t seed, uint32_t* codes, float* scale, float* minv);
void orc_aqsgd_quant_decompress(const uint32_t* codes, const float* scale, const float* minv,
                                float* buf_recv, int64_t num_samples,
                                const int64_t* sample_ids, int64_t n_ids,
                                int64_t rows_per_sample, int64_t row_len, int bits);

#ifdef __cplusplus
}
#endif
#endif
