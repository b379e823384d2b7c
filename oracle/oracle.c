/*
 * oracle.c -- CPU oracle for the compression operators of Rudakov et al.,
 * "Activations and Gradients Compression for Model-Parallel Training"
 * (arXiv 2401.07788).
 *
 * TEST INFRASTRUCTURE ONLY: tests, the smoke check and the CPU-baseline leg of
 * the benchmark call it; the product path never does.  It is plain,
 * single-threaded C written from the paper's definitions; it shares no code
 * with the CUDA library.  Build: -O2 -ffp-contract=off, no fast-math, so every
 * float expression below is one IEEE binary32 round-to-nearest-even operation
 * per operator, evaluated in the order written.
 *
 * Readings of points the paper leaves open (each also listed in the design
 * notes):
 *  - rows: every operator acts on each row of a [rows][row_len] matrix
 *    independently ("input vector", §2.2, §2.3);
 *  - TopK order: magnitude descending, equal magnitudes by lower index first;
 *    the payload lists the kept entries by ascending index, values keep their
 *    sign bits (§2.3);
 *  - quantisation: 2^bits levels, codes 0 .. 2^bits-1, per-row fp32 min and
 *    scale, min and max taken in the total order with -0 < +0 (§2.2);
 *  - stochastic rounding and its counter-based generator are not in the paper.
 *
 * Parity status: no function here has a worked numerical example in the paper
 * (it prints none).  Each is pinned instead by closed forms, invariants,
 * published generator outputs and brute force (tests/test_oracle_pins.py).
 */
#include "oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------- */
/* Counter-based generator (not in the paper).                               */
/* ------------------------------------------------------------------------- */

/* splitmix64: Steele, Lea & Flood, "Fast splittable pseudorandom number
 * generators", OOPSLA 2014.  The generator's state after c+1 steps from seed
 * is seed + (c+1)*GAMMA; its output is the variant-13 finaliser of that state. */
uint64_t orc_splitmix64(uint64_t seed, uint64_t counter)
{
    const uint64_t GAMMA = 0x9E3779B97F4A7C15ull;
    uint64_t z = seed + (counter + 1u) * GAMMA;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

float orc_uniform(uint64_t seed, uint64_t i)
{
    uint64_t z = orc_splitmix64(seed, i >> 1);
    uint32_t half = (i & 1u) ? (uint32_t)(z >> 32) : (uint32_t)(z & 0xffffffffu);
    /* 24 random bits scaled by 2^-24: exact in binary32, u in [0, 1). */
    return (float)(half >> 8) * 0x1p-24f;
}

/* ------------------------------------------------------------------------- */
/* TopK, §2.3                                                                */
/* ------------------------------------------------------------------------- */

typedef struct {
    float mag;  /* |x_j| */
    int64_t j;  /* column index */
} orc_entry;

/* "largest K% values (in absolute value)": larger magnitude first; equal
 * magnitudes are ordered by lower index first. */
static int by_magnitude_desc(const void* pa, const void* pb)
{
    const orc_entry* a = (const orc_entry*)pa;
    const orc_entry* b = (const orc_entry*)pb;
    if (a->mag > b->mag) return -1;
    if (a->mag < b->mag) return 1;
    return (a->j < b->j) ? -1 : (a->j > b->j);
}

static int by_index_asc(const void* pa, const void* pb)
{
    const orc_entry* a = (const orc_entry*)pa;
    const orc_entry* b = (const orc_entry*)pb;
    return (a->j < b->j) ? -1 : (a->j > b->j);
}

/* One row: sort every entry by magnitude, keep the first k, list them by
 * ascending index with their original (signed) values. */
static void topk_row(const float* x, int64_t row_len, int64_t k, float* vals,
                     int32_t* idx, orc_entry* work)
{
    for (int64_t j = 0; j < row_len; ++j) {
        work[j].mag = fabsf(x[j]);
        work[j].j = j;
    }
    qsort(work, (size_t)row_len, sizeof(orc_entry), by_magnitude_desc);
    qsort(work, (size_t)k, sizeof(orc_entry), by_index_asc);
    for (int64_t i = 0; i < k; ++i) {
        idx[i] = (int32_t)work[i].j;
        vals[i] = x[work[i].j];
    }
}

void orc_topk_compress(const float* x, int64_t rows, int64_t row_len, int64_t k,
                       float* vals, int32_t* idx)
{
    orc_entry* work = (orc_entry*)malloc(sizeof(orc_entry) * (size_t)row_len);
    for (int64_t r = 0; r < rows; ++r)
        topk_row(x + r * row_len, row_len, k, vals + r * k, idx + r * k, work);
    free(work);
}

/* Decompression (§2.3): a dense row of +0 with the kept values put back at
 * their indices. */
void orc_topk_decompress(const float* vals, const int32_t* idx, int64_t rows,
                         int64_t row_len, int64_t k, float* y)
{
    for (int64_t r = 0; r < rows; ++r) {
        float* yr = y + r * row_len;
        for (int64_t j = 0; j < row_len; ++j) yr[j] = 0.0f;
        for (int64_t i = 0; i < k; ++i) yr[idx[r * k + i]] = vals[r * k + i];
    }
}

/* TopK index reuse, §3.2 (Table 5): the gradient at a boundary is compressed
 * at the indices kept for the activation in the forward pass, so the payload
 * is the gradient's values at those indices, in the same order. */
void orc_topk_gather(const float* g, int64_t rows, int64_t row_len, const int32_t* idx,
                     int64_t k, float* vals)
{
    for (int64_t r = 0; r < rows; ++r)
        for (int64_t i = 0; i < k; ++i)
            vals[r * k + i] = g[r * row_len + idx[r * k + i]];
}

/* ------------------------------------------------------------------------- */
/* Error feedback (Seide et al.), §2.4                                        */
/* ------------------------------------------------------------------------- */

/* The message is C(X + e); the error left behind is e' = s - C(s) with
 * s = X + e.  The buffer e is global: one per operator, carried across calls. */
void orc_ef_topk_compress(const float* x, float* e, int64_t rows, int64_t row_len,
                          int64_t k, float* vals, int32_t* idx)
{
    float* s = (float*)malloc(sizeof(float) * (size_t)row_len);
    float* c = (float*)malloc(sizeof(float) * (size_t)row_len);
    orc_entry* work = (orc_entry*)malloc(sizeof(orc_entry) * (size_t)row_len);
    for (int64_t r = 0; r < rows; ++r) {
        const float* xr = x + r * row_len;
        float* er = e + r * row_len;
        for (int64_t j = 0; j < row_len; ++j) s[j] = xr[j] + er[j];
        topk_row(s, row_len, k, vals + r * k, idx + r * k, work);
        orc_topk_decompress(vals + r * k, idx + r * k, 1, row_len, k, c);
        for (int64_t j = 0; j < row_len; ++j) er[j] = s[j] - c[j];
    }
    free(work);
    free(c);
    free(s);
}

/* ------------------------------------------------------------------------- */
/* EF21 (Richtarik et al.), §2.4, and AQ-SGD (Wang et al.), §2.5              */
/* ------------------------------------------------------------------------- */

/* One row of the EF21 step: the message is C(X - g) and g' = g + C(X - g).
 * C(X - g) is zero off its support, and adding zero leaves g as it was, so
 * only the kept entries of g change (their sign-of-zero bits included). */
static void delta_row(const float* xr, float* gr, int64_t row_len, int64_t k,
                      float* vals, int32_t* idx, float* d, orc_entry* work)
{
    for (int64_t j = 0; j < row_len; ++j) d[j] = xr[j] - gr[j];
    topk_row(d, row_len, k, vals, idx, work);
    for (int64_t i = 0; i < k; ++i) gr[idx[i]] = gr[idx[i]] + vals[i];
}

/* EF-mixed, §2.4: the k largest magnitudes are split between the input and the
 * error buffer, half each, and x + e is sent on the chosen entries.  Reading:
 * the input's share is its ceil(k/2) largest |x|; the buffer's share, its
 * floor(k/2) largest |e| among the entries the input's share did not take, so
 * that exactly k entries are sent as the section states; the buffer keeps
 * x + e everywhere else (e <- s - C(s) as in error feedback). */
void orc_efmix_topk_compress(const float* x, float* e, int64_t rows, int64_t row_len,
                             int64_t k, float* vals, int32_t* idx)
{
    const int64_t k1 = k - k / 2, k2 = k / 2;
    orc_entry* work = (orc_entry*)malloc(sizeof(orc_entry) * (size_t)row_len);
    char* taken = (char*)malloc((size_t)row_len);
    for (int64_t r = 0; r < rows; ++r) {
        const float* xr = x + r * row_len;
        float* er = e + r * row_len;
        memset(taken, 0, (size_t)row_len);
        /* the input's share */
        for (int64_t j = 0; j < row_len; ++j) {
            work[j].mag = fabsf(xr[j]);
            work[j].j = j;
        }
        qsort(work, (size_t)row_len, sizeof(orc_entry), by_magnitude_desc);
        for (int64_t i = 0; i < k1; ++i) taken[work[i].j] = 1;
        /* the buffer's share, among the entries left */
        int64_t m = 0;
        for (int64_t j = 0; j < row_len; ++j)
            if (!taken[j]) {
                work[m].mag = fabsf(er[j]);
                work[m].j = j;
                ++m;
            }
        qsort(work, (size_t)m, sizeof(orc_entry), by_magnitude_desc);
        for (int64_t i = 0; i < k2; ++i) taken[work[i].j] = 1;
        /* send s = x + e on the chosen entries, keep it elsewhere */
        int64_t n = 0;
        for (int64_t j = 0; j < row_len; ++j) {
            float sj = xr[j] + er[j];
            if (taken[j]) {
                idx[r * k + n] = (int32_t)j;
                vals[r * k + n] = sj;
                ++n;
                er[j] = 0.0f;
            } else {
                er[j] = sj;
            }
        }
    }
    free(taken);
    free(work);
}

void orc_ef21_topk_compress(const float* x, float* g, int64_t rows, int64_t row_len,
                            int64_t k, float* vals, int32_t* idx)
{
    float* d = (float*)malloc(sizeof(float) * (size_t)row_len);
    orc_entry* work = (orc_entry*)malloc(sizeof(orc_entry) * (size_t)row_len);
    for (int64_t r = 0; r < rows; ++r)
        delta_row(x + r * row_len, g + r * row_len, row_len, k, vals + r * k,
                  idx + r * k, d, work);
    free(work);
    free(d);
}

/* AQ-SGD keeps one buffer per training sample: for the i-th listed sample the
 * change X - buf[id] is compressed and buf[id] takes the compressed change.
 * Logical row i*rows_per_sample + r of x and of the payload belongs to row r
 * of sample sample_ids[i]; ids are processed in the order listed. */
void orc_aqsgd_compress(const float* x, float* buf, int64_t num_samples,
                        const int64_t* sample_ids, int64_t n_ids,
                        int64_t rows_per_sample, int64_t row_len, int64_t k,
                        float* vals, int32_t* idx)
{
    (void)num_samples;
    float* d = (float*)malloc(sizeof(float) * (size_t)row_len);
    orc_entry* work = (orc_entry*)malloc(sizeof(orc_entry) * (size_t)row_len);
    for (int64_t i = 0; i < n_ids; ++i) {
        for (int64_t r = 0; r < rows_per_sample; ++r) {
            int64_t logical = i * rows_per_sample + r;
            int64_t stored = sample_ids[i] * rows_per_sample + r;
            delta_row(x + logical * row_len, buf + stored * row_len, row_len, k,
                      vals + logical * k, idx + logical * k, d, work);
        }
    }
    free(work);
    free(d);
}

/* Receiver side: its own copy of the per-sample buffer takes the same update
 * buf[id] <- buf[id] + decompress(payload). */
void orc_aqsgd_decompress(const float* vals, const int32_t* idx, float* buf_recv,
                          int64_t num_samples, const int64_t* sample_ids,
                          int64_t n_ids, int64_t rows_per_sample, int64_t row_len,
                          int64_t k)
{
    (void)num_samples;
    for (int64_t i = 0; i < n_ids; ++i) {
        for (int64_t r = 0; r < rows_per_sample; ++r) {
            int64_t logical = i * rows_per_sample + r;
            float* br = buf_recv + (sample_ids[i] * rows_per_sample + r) * row_len;
            for (int64_t t = 0; t < k; ++t) {
                int32_t j = idx[logical * k + t];
                br[j] = br[j] + vals[logical * k + t];
            }
        }
    }
}

/* ------------------------------------------------------------------------- */
/* Min-max quantisation, §2.2                                                */
/* ------------------------------------------------------------------------- */

/* Total order on finite floats in which -0 sorts below +0. */
static int total_less(float a, float b)
{
    if (a < b) return 1;
    if (a > b) return 0;
    return signbit(a) && !signbit(b);
}

int64_t orc_quant_row_words(int64_t row_len, int bits)
{
    int64_t words = (row_len * (int64_t)bits + 31) / 32;
    return (words + 3) / 4 * 4; /* rows start on 16-byte boundaries */
}

/* Code j of a row occupies bits [j*bits, j*bits + bits) of the row's
 * bitstream; bit p of the stream is bit p%32 of word p/32. */
static void put_code(uint32_t* row_codes, int64_t j, int bits, uint32_t q)
{
    int64_t p = j * (int64_t)bits;
    int64_t w = p >> 5;
    int off = (int)(p & 31);
    row_codes[w] |= q << off;
    if (off + bits > 32) row_codes[w + 1] |= q >> (32 - off);
}

static uint32_t get_code(const uint32_t* row_codes, int64_t j, int bits)
{
    int64_t p = j * (int64_t)bits;
    int64_t w = p >> 5;
    int off = (int)(p & 31);
    uint64_t both = (uint64_t)row_codes[w] >> off;
    if (off + bits > 32) both |= (uint64_t)row_codes[w + 1] << (32 - off);
    return (uint32_t)(both & ((1ull << bits) - 1u));
}

/* §2.2: each row is shifted by its minimum and divided by its range, which
 * puts it in [0, 1], and then rounded onto 2^bits evenly spaced levels; with
 * L = 2^bits - 1 intervals,
 *   scale = (max - min) / L,  inv = L / (max - min),
 *   t = (x - min) * inv,  q = round(t)  or  floor(t + u),  clamped to [0, L].
 * A row whose range is 0, or whose range or inv is infinite, sends all-zero
 * codes with scale 0 and min = its minimum. */
void orc_quant_compress(const float* x, int64_t rows, int64_t row_len, int bits,
                        int mode, uint64_t seed, uint32_t* codes, float* scale,
                        float* minv)
{
    int64_t W = orc_quant_row_words(row_len, bits);
    for (int64_t r = 0; r < rows; ++r) {
        const float* xr = x + r * row_len;
        uint32_t* cr = codes + r * W;
        memset(cr, 0, sizeof(uint32_t) * (size_t)W);
        if (bits == 32) { /* passthrough: raw binary32 bits */
            memcpy(cr, xr, sizeof(float) * (size_t)row_len);
            scale[r] = 0.0f;
            minv[r] = 0.0f;
            continue;
        }
        float mn = xr[0], mx = xr[0];
        for (int64_t j = 1; j < row_len; ++j) {
            if (total_less(xr[j], mn)) mn = xr[j];
            if (total_less(mx, xr[j])) mx = xr[j];
        }
        float levels = (float)((1u << bits) - 1u);
        float range = mx - mn;
        float inv = levels / range;
        int degenerate = (range == 0.0f) || isinf(range) || isinf(inv);
        scale[r] = degenerate ? 0.0f : range / levels;
        minv[r] = mn;
        if (degenerate) continue;
        for (int64_t j = 0; j < row_len; ++j) {
            float t = (xr[j] - mn) * inv;
            float qf;
            if (mode == 0) {
                qf = rintf(t); /* nearest, ties to even */
            } else {
                float u = orc_uniform(seed, (uint64_t)(r * row_len + j));
                qf = floorf(t + u);
            }
            if (qf < 0.0f) qf = 0.0f;
            if (qf > levels) qf = levels;
            put_code(cr, j, bits, (uint32_t)qf);
        }
    }
}

/* Decompression (§2.2), the codes mapped back to the row's range:
 * y = min + q * scale. */
void orc_quant_decompress(const uint32_t* codes, const float* scale, const float* minv,
                          int64_t rows, int64_t row_len, int bits, float* y)
{
    int64_t W = orc_quant_row_words(row_len, bits);
    for (int64_t r = 0; r < rows; ++r) {
        const uint32_t* cr = codes + r * W;
        float* yr = y + r * row_len;
        if (bits == 32) {
            memcpy(yr, cr, sizeof(float) * (size_t)row_len);
            continue;
        }
        for (int64_t j = 0; j < row_len; ++j) {
            float q = (float)get_code(cr, j, bits);
            yr[j] = minv[r] + q * scale[r];
        }
    }
}

/* AQ-SGD with quantisation, §2.5 (the cited work compresses the change of the
 * activations by quantisation; the section applies the same scheme with
 * TopK): for each listed sample id and row, d = x - buf[id, r], the message is
 * Quant(d) (§2.2, the quantiser above on the gathered rows, logical row i * rps
 * + r), and buf[id, r] <- buf[id, r] + Dequant(Quant(d)). */
void orc_aqsgd_quant_compress(const float* x, float* buf, int64_t num_samples,
                              const int64_t* sample_ids, int64_t n_ids,
                              int64_t rows_per_sample, int64_t row_len, int bits, int mode,
                              uint64_t seed, uint32_t* codes, float* scale, float* minv)
{
    (void)num_samples;
    const int64_t rows = n_ids * rows_per_sample;
    float* d = (float*)malloc(sizeof(float) * (size_t)(rows * row_len));
    float* dh = (float*)malloc(sizeof(float) * (size_t)(rows * row_len));
    for (int64_t i = 0; i < n_ids; ++i)
        for (int64_t r = 0; r < rows_per_sample; ++r) {
            const int64_t logical = i * rows_per_sample + r;
            const float* br = buf + (sample_ids[i] * rows_per_sample + r) * row_len;
            for (int64_t j = 0; j < row_len; ++j)
                d[logical * row_len + j] = x[logical * row_len + j] - br[j];
        }
    orc_quant_compress(d, rows, row_len, bits, mode, seed, codes, scale, minv);
    orc_quant_decompress(codes, scale, minv, rows, row_len, bits, dh);
    for (int64_t i = 0; i < n_ids; ++i)
        for (int64_t r = 0; r < rows_per_sample; ++r) {
            const int64_t logical = i * rows_per_sample + r;
            float* br = buf + (sample_ids[i] * rows_per_sample + r) * row_len;
            for (int64_t j = 0; j < row_len; ++j) br[j] = br[j] + dh[logical * row_len + j];
        }
    free(dh);
    free(d);
}

/* The receiver's side: buf_recv[id, r] <- buf_recv[id, r] + Dequant(codes of the
 * logical row), which it then uses as the activation. */
void orc_aqsgd_quant_decompress(const uint32_t* codes, const float* scale, const float* minv,
                                float* buf_recv, int64_t num_samples,
                                const int64_t* sample_ids, int64_t n_ids,
                                int64_t rows_per_sample, int64_t row_len, int bits)
{
    (void)num_samples;
    const int64_t rows = n_ids * rows_per_sample;
    float* dh = (float*)malloc(sizeof(float) * (size_t)(rows * row_len));
    orc_quant_decompress(codes, scale, minv, rows, row_len, bits, dh);
    for (int64_t i = 0; i < n_ids; ++i)
        for (int64_t r = 0; r < rows_per_sample; ++r) {
            const int64_t logical = i * rows_per_sample + r;
            float* br = buf_recv + (sample_ids[i] * rows_per_sample + r) * row_len;
            for (int64_t j = 0; j < row_len; ++j) br[j] = br[j] + dh[logical * row_len + j];
        }
    free(dh);
}
