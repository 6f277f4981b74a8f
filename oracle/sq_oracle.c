/*
 * Scale-QLoRA reference oracle: a plain, slow, float64 CPU statement of the
 * scale-only training step's hot path.
 *
 * THIS IS TEST INFRASTRUCTURE. Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load it. The CUDA library never calls it and
 * shares no code, table or constant with it.
 *
 * Sources (section / equation names of arXiv 2609.04526):
 *  - Sec. 2 "Native FP4 microscaling storage": W[o,i] = code[o,i] * eff_scale[o, i // block],
 *    E2M1 codes from +-{0,.5,1,1.5,2,3,4,6}; NVFP4 = block 16 with an E4M3 byte
 *    (max 448) times one fp32 tensor scale ws2; MXFP4 = block 32 with an E8M0
 *    power-of-two byte.
 *  - Sec. 3 "Scale-QLoRA forward": y = x W'^T with fp32 scale arithmetic; the
 *    backward (dX, scale gradient) is the derivative of that bilinear form.
 *  - Sec. 3 "QAST makes merge exact by construction": round_grid(s) is
 *    e4m3(s/ws2)*ws2 on NVFP4 and 2^round(log2 s) on MXFP4; merge writes the
 *    on-grid byte and never a code.
 *  - Sec. 3 "A single-setting stability recipe" (ii)/(iii): the E4M3 ceiling
 *    clamp min(eff, 448*ws2), shared by the forward and the merge.
 *  - Sec. 5 "Payoff 3: invertible merges and rollback": the on-grid delta.
 *
 * Readings where the paper is silent (nibble order, lower clamp, E8M0 range,
 * NaN handling) follow the repository's design notes and are repeated at each
 * function below.
 *
 * Build: gcc -O2 -fopenmp -ffp-contract=off -shared -fPIC (contraction off so the
 * fp32 steps of the projection and merge are the plain IEEE operations written).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define OR_NVFP4 0
#define OR_MXFP4 1

/* ------------------------------------------------------------------ */
/* Format decode (Sec. 2, OCP MX / NVFP4 definitions)                   */
/* ------------------------------------------------------------------ */

/* E2M1: 1 sign bit, 2 exponent bits (bias 1), 1 mantissa bit, no inf/NaN.
 * exponent field 0 is subnormal: 0.5 * m. Gives +-{0,.5,1,1.5,2,3,4,6}. */
double or_e2m1(int nibble) {
    int s = (nibble >> 3) & 1, e = (nibble >> 1) & 3, m = nibble & 1;
    double mag = (e == 0) ? 0.5 * m : ldexp(1.0 + 0.5 * m, e - 1);
    return s ? -mag : mag;
}

/* E4M3 "fn": 1 sign, 4 exponent bits (bias 7), 3 mantissa bits; no inf; only
 * S.1111.111 is NaN, so the largest finite value is 448 (Sec. 2). */
double or_e4m3(int byte) {
    int s = (byte >> 7) & 1, e = (byte >> 3) & 15, m = byte & 7;
    double mag;
    if (e == 15 && m == 7) return NAN;
    if (e == 0) mag = ldexp((double)m, -9);            /* m/8 * 2^(1-7) */
    else mag = ldexp(1.0 + m / 8.0, e - 7);
    return s ? -mag : mag;
}

/* E8M0: unsigned exponent byte, bias 127, no mantissa, no zero; 255 is NaN. */
double or_e8m0(int byte) {
    if (byte == 255) return NAN;
    return ldexp(1.0, byte - 127);
}

/* Element k of code row n. Layout reading: codes are [N, K/2] bytes, two
 * codes per byte, the even k in the low nibble. */
int or_code_nibble(const uint8_t *codes, int64_t K, int64_t n, int64_t k) {
    uint8_t byte = codes[n * (K / 2) + k / 2];
    return (k & 1) ? (byte >> 4) : (byte & 15);
}

int or_block(int fmt) { return fmt == OR_NVFP4 ? 16 : 32; }

/* Effective block scale eff_scale[n,b] (Sec. 2): E4M3(byte)*ws2 or E8M0(byte).
 * The product of a 4-bit and a 24-bit significand is exact in float64. */
double or_eff_scale(int fmt, const uint8_t *scales, int64_t G, float ws2, int64_t n, int64_t b) {
    int byte = scales[n * G + b];
    return fmt == OR_NVFP4 ? or_e4m3(byte) * (double)ws2 : or_e8m0(byte);
}

/* W[n,k] = code[n,k] * eff_scale[n, k // block] (Sec. 2), into a float64 [N,K]. */
void or_decode_weight(int fmt, int64_t N, int64_t K, const uint8_t *codes, const uint8_t *scales,
                      float ws2, double *W) {
    int64_t B = or_block(fmt), G = K / B;
    for (int64_t n = 0; n < N; n++)
        for (int64_t k = 0; k < K; k++)
            W[n * K + k] = or_e2m1(or_code_nibble(codes, K, n, k)) * or_eff_scale(fmt, scales, G, ws2, n, k / B);
}

/* bf16 -> float64: a bf16 is the top half of an fp32. */
double or_bf16(uint16_t h) {
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, 4);
    return (double)f;
}

static double *bf16_to_f64(const uint16_t *x, int64_t count) {
    double *d = (double *)malloc(sizeof(double) * (size_t)(count > 0 ? count : 1));
    for (int64_t i = 0; i < count; i++) d[i] = or_bf16(x[i]);
    return d;
}

/* ------------------------------------------------------------------ */
/* Contractions on float64 operands (Sec. 3 forward and its backward)   */
/* ------------------------------------------------------------------ */

/* Y[m,n] = sum_k X[m,k] W[n,k]  (y = x W'^T). */
void or_fwd_f64(int64_t M, int64_t N, int64_t K, const double *X, const double *W, double *Y) {
#pragma omp parallel for schedule(static)
    for (int64_t m = 0; m < M; m++)
        for (int64_t n = 0; n < N; n++) {
            double acc = 0.0;
            for (int64_t k = 0; k < K; k++) acc += X[m * K + k] * W[n * K + k];
            Y[m * N + n] = acc;
        }
}

/* dX[m,k] = sum_n dY[m,n] W[n,k]: the input gradient of y = x W^T. */
void or_dx_f64(int64_t M, int64_t N, int64_t K, const double *dY, const double *W, double *dX) {
#pragma omp parallel for schedule(static)
    for (int64_t m = 0; m < M; m++) {
        double *row = dX + m * K;
        for (int64_t k = 0; k < K; k++) row[k] = 0.0;
        for (int64_t n = 0; n < N; n++) {
            double d = dY[m * N + n];
            for (int64_t k = 0; k < K; k++) row[k] += d * W[n * K + k];
        }
    }
}

/* Scale gradient with respect to the effective scale (absolute units):
 *   D[n,k]  = sum_m dY[m,n] X[m,k]            (the weight gradient dW = dY^T X)
 *   g[n,b]  = sum_{k in block b} code[n,k] D[n,k]
 * since dW[n,k] = code[n,k] * d eff_scale[n, k//B] (Sec. 3 forward).  If mask is
 * given, g[n,b] is multiplied by mask[n,b] (the STE pass-through of the clamp,
 * Sec. 3 stability recipe (ii)). Rows listed in `rows` only (all rows if rows is NULL). */
void or_scale_grad_f64(int64_t M, int64_t N, int64_t K, int B, const uint8_t *codes, const double *X,
                       const double *dY, const uint8_t *mask, int64_t nrows, const int64_t *rows,
                       double *g /* [nrows or N, K/B] */) {
    int64_t G = K / B;
    int64_t R = rows ? nrows : N;
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t r = 0; r < R; r++) {
        int64_t n = rows ? rows[r] : r;
        double *D = (double *)calloc((size_t)(K > 0 ? K : 1), sizeof(double));
        for (int64_t m = 0; m < M; m++) {
            double d = dY[m * N + n];
            for (int64_t k = 0; k < K; k++) D[k] += d * X[m * K + k];
        }
        for (int64_t b = 0; b < G; b++) {
            double acc = 0.0;
            for (int64_t k = b * B; k < (b + 1) * B; k++) acc += or_e2m1(or_code_nibble(codes, K, n, k)) * D[k];
            if (mask) acc *= (double)mask[n * G + b];
            g[r * G + b] = acc;
        }
        free(D);
    }
}

/* ------------------------------------------------------------------ */
/* Entry points on the packed formats                                   */
/* ------------------------------------------------------------------ */

void or_fwd(int fmt, int64_t N, int64_t K, const uint8_t *codes, const uint8_t *scales, float ws2,
            int64_t M, const uint16_t *X_bf16, double *Y) {
    double *W = (double *)malloc(sizeof(double) * (size_t)(N * K));
    double *X = bf16_to_f64(X_bf16, M * K);
    or_decode_weight(fmt, N, K, codes, scales, ws2, W);
    or_fwd_f64(M, N, K, X, W, Y);
    free(W);
    free(X);
}

void or_dx(int fmt, int64_t N, int64_t K, const uint8_t *codes, const uint8_t *scales, float ws2,
           int64_t M, const uint16_t *dY_bf16, double *dX) {
    double *W = (double *)malloc(sizeof(double) * (size_t)(N * K));
    double *dY = bf16_to_f64(dY_bf16, M * N);
    or_decode_weight(fmt, N, K, codes, scales, ws2, W);
    or_dx_f64(M, N, K, dY, W, dX);
    free(W);
    free(dY);
}

void or_scale_grad(int fmt, int64_t N, int64_t K, const uint8_t *codes, int64_t M, const uint16_t *X_bf16,
                   const uint16_t *dY_bf16, const uint8_t *mask, int64_t nrows, const int64_t *rows, double *g) {
    double *X = bf16_to_f64(X_bf16, M * K);
    double *dY = bf16_to_f64(dY_bf16, M * N);
    or_scale_grad_f64(M, N, K, or_block(fmt), codes, X, dY, mask, nrows, rows, g);
    free(X);
    free(dY);
}

/* Sampled forward: out[i] = Y[ms[i], ns[i]], one dot product per sample. */
void or_fwd_at(int fmt, int64_t N, int64_t K, const uint8_t *codes, const uint8_t *scales, float ws2,
               int64_t M, const uint16_t *X_bf16, int64_t count, const int64_t *ms, const int64_t *ns,
               double *out) {
    int64_t B = or_block(fmt), G = K / B;
    (void)M;
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < count; i++) {
        int64_t m = ms[i], n = ns[i];
        double acc = 0.0;
        for (int64_t k = 0; k < K; k++)
            acc += or_bf16(X_bf16[m * K + k]) * or_e2m1(or_code_nibble(codes, K, n, k)) *
                   or_eff_scale(fmt, scales, G, ws2, n, k / B);
        out[i] = acc;
    }
}

/* Sampled input gradient: out[i] = dX[ms[i], ks[i]]. */
void or_dx_at(int fmt, int64_t N, int64_t K, const uint8_t *codes, const uint8_t *scales, float ws2,
              int64_t M, const uint16_t *dY_bf16, int64_t count, const int64_t *ms, const int64_t *ks,
              double *out) {
    int64_t B = or_block(fmt), G = K / B;
    (void)M;
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < count; i++) {
        int64_t m = ms[i], k = ks[i];
        double acc = 0.0;
        for (int64_t n = 0; n < N; n++)
            acc += or_bf16(dY_bf16[m * N + n]) * or_e2m1(or_code_nibble(codes, K, n, k)) *
                   or_eff_scale(fmt, scales, G, ws2, n, k / B);
        out[i] = acc;
    }
}

/* ------------------------------------------------------------------ */
/* Grid projection (Sec. 3 QAST round_grid + ceiling clamp)             */
/* ------------------------------------------------------------------ */

/* Nearest finite E4M3 byte to q with ties to the even mantissa; the sign of q
 * (including -0) is kept. Every finite magnitude 0x00..0x7E is a candidate, so
 * values past 448 land on 448. Distances are float64 differences: for an fp32
 * q the two candidates that bracket it subtract exactly (Sterbenz, or a span of
 * under 53 bits), so the winner and any tie are decided exactly. */
int or_e4m3_rne(float q) {
    double a = fabs((double)q);
    int best = 0;
    double bestd = INFINITY;
    for (int c = 0; c <= 0x7E; c++) {
        double d = fabs(a - or_e4m3(c));
        if (d < bestd || (d == bestd && (c & 1) == 0 && (best & 1) == 1)) {
            best = c;
            bestd = d;
        }
    }
    return signbit(q) ? (best | 0x80) : best;
}

/* round(log2 L) for a finite L > 0, evaluated exactly: L = m * 2^E with m in
 * [1,2); round up iff m > sqrt(2), i.e. m*m > 2 (m has 24 significant bits so
 * m*m is exact in float64). The midpoint is the geometric one of the formula
 * 2^round(log2 s); fp32 inputs never tie because sqrt(2) is irrational. */
int or_round_log2(float L) {
    int x;
    double f = frexp((double)L, &x); /* L = f * 2^x, f in [0.5, 1) */
    double m = 2.0 * f;
    int E = x - 1;
    return E + ((m * m > 2.0) ? 1 : 0);
}

/* Project one latent scale L (absolute units) onto the grid.
 * NVFP4: cap = fl32(448*ws2); q = fl32(clamp(L, -cap, cap) / ws2); byte = RNE-E4M3(q).
 *        mask = 1 iff -cap <= L <= cap (the clamp passes the gradient at equality).
 *        NaN -> 0x7F, mask 0, counted. The lower saturation at -cap is this
 *        build's reading (the paper states only the ceiling).
 * MXFP4: byte = round(log2 L) + 127 clamped to [0, 254]; mask 0 when clamped;
 *        L <= 0 (no sign or zero in E8M0) -> byte 0, mask 0; +inf -> 254, mask 0;
 *        NaN -> 0xFF, mask 0, counted. */
void or_project_one(int fmt, float ws2, float L, uint8_t *byte, uint8_t *mask, int *is_nan) {
    *is_nan = 0;
    if (isnan(L)) {
        *byte = fmt == OR_NVFP4 ? 0x7F : 0xFF;
        *mask = 0;
        *is_nan = 1;
        return;
    }
    if (fmt == OR_NVFP4) {
        float cap = 448.0f * ws2;
        float Lc = L;
        if (Lc > cap) Lc = cap;
        if (Lc < -cap) Lc = -cap;
        float q = Lc / ws2;
        *byte = (uint8_t)or_e4m3_rne(q);
        *mask = (L >= -cap && L <= cap) ? 1 : 0;
    } else {
        if (!(L > 0.0f)) {
            *byte = 0;
            *mask = 0;
            return;
        }
        if (isinf(L)) {
            *byte = 254;
            *mask = 0;
            return;
        }
        int e = or_round_log2(L) + 127;
        *mask = 1;
        if (e < 0) { e = 0; *mask = 0; }
        if (e > 254) { e = 254; *mask = 0; }
        *byte = (uint8_t)e;
    }
}

/* Projection of a whole [N, G] plane (row-major, treated as count = N*G values). */
void or_project(int fmt, int64_t count, float ws2, const float *latent, uint8_t *bytes, uint8_t *mask,
                int64_t *nonfinite) {
    int64_t nan_count = 0;
    for (int64_t i = 0; i < count; i++) {
        uint8_t b, mk;
        int isn;
        or_project_one(fmt, ws2, latent[i], &b, &mk, &isn);
        bytes[i] = b;
        if (mask) mask[i] = mk;
        nan_count += isn;
    }
    if (nonfinite) *nonfinite = nan_count;
}

/* Decoded scale of a byte in fp32: E4M3(byte)*ws2 (one fp32 multiply) or E8M0(byte). */
float or_scale_f32(int fmt, float ws2, uint8_t byte) {
    if (fmt == OR_NVFP4) return (float)or_e4m3(byte) * ws2;
    return (float)or_e8m0(byte);
}

/* Merge (Sec. 3: merge writes exactly the on-grid scale byte the forward used
 * and never a code): scales_inout <- projection(latent). No code plane is an
 * argument. Optional on-grid delta in fp32, delta = fl32(s(new) - s(old)), the
 * quantity whose subtraction restores the base (Sec. 5, Payoff 3). changed =
 * number of bytes that differ. */
void or_merge(int fmt, int64_t count, float ws2, const float *latent, uint8_t *scales_inout, float *delta,
              int64_t *changed) {
    int64_t ch = 0;
    for (int64_t i = 0; i < count; i++) {
        uint8_t b, mk;
        int isn;
        uint8_t old = scales_inout[i];
        or_project_one(fmt, ws2, latent[i], &b, &mk, &isn);
        if (delta) {
            float sn = or_scale_f32(fmt, ws2, b);
            float so = or_scale_f32(fmt, ws2, old);
            delta[i] = sn - so;
        }
        ch += (b != old);
        scales_inout[i] = b;
    }
    if (changed) *changed = ch;
}

/* Rollback (Sec. 5, Payoff 3: subtracting the on-grid scale delta the merge
 * applied restores the base checkpoint byte for byte): every byte is replaced by
 * the projection (same grid and clamp path as the merge) of fl32(s(byte) - delta)
 * with s(byte) as or_scale_f32. changed = number of bytes that differ. */
void or_rollback(int fmt, int64_t count, float ws2, const float *delta, uint8_t *scales_inout, int64_t *changed) {
    int64_t ch = 0;
    for (int64_t i = 0; i < count; i++) {
        uint8_t b, mk;
        int isn;
        const uint8_t old = scales_inout[i];
        const float back = or_scale_f32(fmt, ws2, old) - delta[i];
        or_project_one(fmt, ws2, back, &b, &mk, &isn);
        ch += (b != old);
        scales_inout[i] = b;
    }
    if (changed) *changed = ch;
}

/* Scale-only hot-swap (Sec. 5 "Hot-swap"): the served task changes by overwriting
 * the scale plane with another adapter's on-grid bytes; no code plane is an
 * argument. changed = number of bytes that differ from the old plane. */
void or_swap(int64_t count, const uint8_t *src, uint8_t *dst, int64_t *changed) {
    int64_t ch = 0;
    for (int64_t i = 0; i < count; i++) {
        ch += (src[i] != dst[i]);
        dst[i] = src[i];
    }
    if (changed) *changed = ch;
}

/* Byte-level audit (Sec. 5): the number of positions where two byte buffers differ. */
int64_t or_count_diff(int64_t count, const uint8_t *a, const uint8_t *b) {
    int64_t d = 0;
    for (int64_t i = 0; i < count; i++) d += (a[i] != b[i]);
    return d;
}

/* ------------------------------------------------------------------ */
/* Low-rank scale adapter (Sec. 3 "Scale-QLoRA forward")                */
/* ------------------------------------------------------------------ */

/* Latent scale of block (n, b): eff'[n,b] = eff[n,b] + (alpha/r) (B A)[n,b], with
 * B [N, r] and A [r, G] bf16 (the paper's trainable factors) and the scale
 * arithmetic in fp32. The paper does not fix the order of the r-term sum; the
 * reading used on both sides: eff = fl32(decode(base byte) * ws2) (or_scale_f32),
 * acc = fp32 fused multiply-adds over j = 0 .. r-1 starting from 0, and
 * eff' = fma(alpha/r, acc, eff) in fp32. Brow = &B[n*r], A is the whole [r, G]. */
float or_lowrank_latent(int fmt, float ws2, float alpha_over_r, int r, uint8_t base_byte, const uint16_t *Brow,
                        const uint16_t *A, int64_t G, int64_t b) {
    float acc = 0.0f;
    for (int j = 0; j < r; j++) acc = fmaf((float)or_bf16(Brow[j]), (float)or_bf16(A[(int64_t)j * G + b]), acc);
    return fmaf(alpha_over_r, acc, or_scale_f32(fmt, ws2, base_byte));
}

/* Projection of the adapter's latent (the grid rounding of the QAST forward,
 * Sec. 3): for every block, eff' as above, then or_project_one. latent (nullable)
 * receives eff' in fp32; nonfinite (nullable) the NaN count. */
void or_project_lowrank(int fmt, int64_t N, int64_t G, int r, float ws2, float alpha_over_r, const uint8_t *base,
                        const uint16_t *B, const uint16_t *A, uint8_t *bytes, uint8_t *mask, int *nonfinite,
                        float *latent) {
    int nan_count = 0;
    for (int64_t n = 0; n < N; n++) {
        for (int64_t b = 0; b < G; b++) {
            const int64_t i = n * G + b;
            const float L = or_lowrank_latent(fmt, ws2, alpha_over_r, r, base[i], B + n * r, A, G, b);
            uint8_t by, mk;
            int isn;
            or_project_one(fmt, ws2, L, &by, &mk, &isn);
            bytes[i] = by;
            if (mask) mask[i] = mk;
            if (latent) latent[i] = L;
            nan_count += isn;
        }
    }
    if (nonfinite) *nonfinite = nan_count;
}

/* Gradients of the adapter factors (Sec. 3: the gradient reaches eff' through the
 * STE, masked by the ceiling clamp, and eff' is linear in B and in A): with gm the
 * masked scale gradient [N, G],
 *   dB[n,j] = (alpha/r) sum_b gm[n,b] A[j,b],   dA[j,b] = (alpha/r) sum_n B[n,j] gm[n,b],
 * in float64. */
void or_lowrank_grad(int64_t N, int64_t G, int r, double alpha_over_r, const float *gm, const uint16_t *B,
                     const uint16_t *A, double *dB, double *dA) {
#pragma omp parallel for schedule(static)
    for (int64_t n = 0; n < N; n++) {
        for (int j = 0; j < r; j++) {
            double s = 0.0;
            for (int64_t b = 0; b < G; b++) s += (double)gm[n * G + b] * or_bf16(A[(int64_t)j * G + b]);
            dB[n * r + j] = alpha_over_r * s;
        }
    }
#pragma omp parallel for schedule(static)
    for (int64_t b = 0; b < G; b++) {
        for (int j = 0; j < r; j++) {
            double s = 0.0;
            for (int64_t n = 0; n < N; n++) s += or_bf16(B[n * r + j]) * (double)gm[n * G + b];
            dA[(int64_t)j * G + b] = alpha_over_r * s;
        }
    }
}

int or_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* ------------------------------------------------------------------ */
/* Scale-family variants (ablation appendix)                           */
/* ------------------------------------------------------------------ */

/* Least-squares code-preserving fit of a weight-space update (the Spider
 * paragraph of the ablations: "solve per block for the least-squares best
 * code-preserving scale delta"). Within block b of row n the representable
 * updates are t * c_b (c_b the block's E2M1 code values), so the fit is
 *   delta[n,b] = <c_b, dW_b> / <c_b, c_b>,
 * in absolute scale units (the update of the block's weights is c_b * delta).
 * Reading: a block whose codes are all zero has no representable direction;
 * its delta is 0. Also returned per block, when the arrays are given:
 *   captured[n,b] = <c_b, dW_b>^2 / <c_b, c_b>   (|| projection ||^2, 0 for a zero block)
 *   total[n,b]    = || dW_b ||^2
 *   latent[n,b]   = fl32(scale(byte) + fl32(delta))   (the fitted scale, for the grid projection)
 * dW is bf16 [N, K]; sums in float64, in element order. */
void or_fit_scale_delta(int fmt, int64_t N, int64_t K, const uint8_t *codes, const uint8_t *scales, float ws2,
                        const uint16_t *dW, double *delta, double *captured, double *total, float *latent) {
  const int B = or_block(fmt);
  const int64_t G = K / B;
#pragma omp parallel for schedule(static)
  for (int64_t n = 0; n < N; ++n) {
    for (int64_t b = 0; b < G; ++b) {
      double cw = 0.0, cc = 0.0, ww = 0.0;
      for (int64_t k = b * B; k < (b + 1) * B; ++k) {
        const double c = or_e2m1(or_code_nibble(codes, K, n, k));
        const double w = or_bf16(dW[n * K + k]);
        cw += c * w;
        cc += c * c;
        ww += w * w;
      }
      const double d = cc > 0.0 ? cw / cc : 0.0;
      delta[n * G + b] = d;
      if (captured) captured[n * G + b] = cc > 0.0 ? cw * cw / cc : 0.0;
      if (total) total[n * G + b] = ww;
      if (latent) latent[n * G + b] = or_scale_f32(fmt, ws2, scales[n * G + b]) + (float)d;
    }
  }
}

/* Granularity ladder (ablations, "Granularity alone over-perturbs"): a direct
 * additive scale delta at granularity gd, one value per group of G / gd
 * consecutive blocks of a row (gd = 1: one per row, PEQA; gd = G: per block).
 * The latent of block b is s(byte) + delta[n, b / (G / gd)], so the gradient of
 * a group delta is the sum of its blocks' (masked) scale gradients:
 *   out[n, j] = sum_{b in group j} g[n, b]            (float64, block order) */
void or_group_reduce(int64_t N, int64_t G, int64_t gd, const float *g, double *out) {
  const int64_t W = G / gd;
  for (int64_t n = 0; n < N; ++n)
    for (int64_t j = 0; j < gd; ++j) {
      double s = 0.0;
      for (int64_t b = j * W; b < (j + 1) * W; ++b) s += (double)g[n * G + b];
      out[n * gd + j] = s;
    }
}

/* Projection of the group-delta latent fl32(s(byte) + delta[n, b / (G / gd)])
 * (one fp32 add, the decoded scale of or_scale_f32) onto the grid. */
void or_project_group_delta(int fmt, int64_t N, int64_t G, int64_t gd, float ws2, const uint8_t *base,
                            const float *delta, uint8_t *bytes, uint8_t *mask, int64_t *nonfinite, float *latent) {
  const int64_t W = G / gd;
  int64_t nan_count = 0;
  for (int64_t n = 0; n < N; ++n)
    for (int64_t b = 0; b < G; ++b) {
      const float L = or_scale_f32(fmt, ws2, base[n * G + b]) + delta[n * gd + b / W];
      int is_nan = 0;
      or_project_one(fmt, ws2, L, &bytes[n * G + b], &mask[n * G + b], &is_nan);
      nan_count += is_nan;
      if (latent) latent[n * G + b] = L;
    }
  *nonfinite = nan_count;
}

/* Full-precision multiplicative control (ablation appendix: unquantized bf16
 * weights, the within-block pattern frozen, one coefficient per (row, block of 16),
 * W' = W (1 + dS[o, g(i)])). Reading of the arithmetic: the factor is
 * f = fl32(1 + dS), the product is rounded to fp32 and then to bf16 (round to
 * nearest, ties to even), i.e. W' = bf16(fl32(W * f)); the contractions then use
 * W' like any decoded weight. */
static float or_round_bf16(float x) {
  uint32_t u;
  memcpy(&u, &x, 4);
  if ((u & 0x7F800000u) == 0x7F800000u) {  /* inf or NaN: keep (quiet NaN) */
    if (u & 0x007FFFFFu) u |= 0x00400000u;
    u &= 0xFFFF0000u;
  } else {
    const uint32_t lsb = (u >> 16) & 1u;
    u = (u + 0x7FFFu + lsb) & 0xFFFF0000u;  /* round half to even at bit 16 */
  }
  float r;
  memcpy(&r, &u, 4);
  return r;
}

void or_control_weight(int64_t N, int64_t K, const uint16_t *W, const float *dS, double *Wp) {
  const int64_t G = K / 16;
  for (int64_t n = 0; n < N; ++n)
    for (int64_t k = 0; k < K; ++k) {
      const float f = 1.0f + dS[n * G + k / 16];
      const float w = (float)or_bf16(W[n * K + k]);
      Wp[n * K + k] = (double)or_round_bf16(w * f);
    }
}

/* Gradient of L with respect to dS[o, b] through W' = W (1 + dS) (the rounding of
 * W' passed straight through): sum over the block's columns of W[o,i] dW[o,i],
 * dW = dY^T X, float64. X [M, K], dY [M, N] as float64. */
void or_control_grad(int64_t M, int64_t N, int64_t K, const uint16_t *W, const double *X, const double *dY,
                     double *g) {
  const int64_t G = K / 16;
#pragma omp parallel for schedule(static)
  for (int64_t n = 0; n < N; ++n)
    for (int64_t b = 0; b < G; ++b) {
      double s = 0.0;
      for (int64_t k = b * 16; k < (b + 1) * 16; ++k) {
        double dw = 0.0;
        for (int64_t m = 0; m < M; ++m) dw += dY[m * N + n] * X[m * K + k];
        s += or_bf16(W[n * K + k]) * dw;
      }
      g[n * G + b] = s;
    }
}

/* The control's low-rank coefficient plane dS = (alpha/r) B A (float64), B [N, r],
 * A [r, G] bf16. */
void or_lowrank_product(int64_t N, int64_t G, int r, double alpha_over_r, const uint16_t *B, const uint16_t *A,
                        double *out) {
  for (int64_t n = 0; n < N; ++n)
    for (int64_t b = 0; b < G; ++b) {
      double s = 0.0;
      for (int j = 0; j < r; ++j) s += or_bf16(B[n * r + j]) * or_bf16(A[(int64_t)j * G + b]);
      out[n * G + b] = alpha_over_r * s;
    }
}
