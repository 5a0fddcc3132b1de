/*
 * ilw_oracle.h -- plain, slow CPU oracle for the integer-only I-LW-DETR forward path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may include, link or call this
 * library: only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference arm
 * use it.  It shares no code, header, table or helper with the CUDA path.
 *
 * Every function is written from the paper ("Enabling Fully Integer-Only Inference for
 * Lightweight Detection Transformers"): Sec. 3.1 (nearest-neighbour deformable sampling, the
 * two-stage pipeline), Sec. 3.2 (integer linear ops, split convolution), Sec. 3.3 (I-LayerNorm,
 * SD-ShiftGELU and I-ViT's ShiftGELU it replaces, Constrained Shiftmax), Table 5 (the detection
 * head's ShiftExp), Algorithm 1 (ShiftExp, SD-ShiftGELU) and Algorithm 2 (CalibrateShift,
 * Constrained Shiftmax).  Where the paper is silent the reading used is stated beside the
 * function.
 *
 * Conventions
 *   - All arithmetic is exact integer arithmetic in int64 (int128 where a product needs it).
 *   - Right shift of a signed value is arithmetic (floor), as C++20 defines it.
 *   - rq(v; m, s) = (v*m + 2^(s-1)) >> s  (dyadic requantisation, round half up; s = 0 -> v*m).
 *   - satN clips to the symmetric range [-(2^(N-1)-1), 2^(N-1)-1] (no zero-point, Sec. 3.2.1).
 *   - Functions return 0 on success and a negative value when an argument is outside the
 *     domain the paper's arithmetic is defined on (e.g. I0 < 1, an overflowing parameter).
 */
#ifndef ILW_ORACLE_H
#define ILW_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Constrained Shiftmax parameters (Algorithm 2 inputs).  s_d < 0 selects the per-row
 * CalibrateShift of Algorithm 2; s_d >= 0 is a static per-module shift (Sec. 3.3.2). */
typedef struct {
    int32_t I0;      /* round(1/S_x) of the score scale (Algorithm 1, ShiftExp) */
    int32_t k_inter; /* intermediate bit precision */
    int32_t k_out;   /* output bit precision */
    int32_t s_d;     /* static denominator shift, or -1 for per-row CalibrateShift */
    int32_t m_p;     /* precision margin (4 in the paper) */
    int32_t M_hw;    /* hardware division precision (31 in the paper) */
} orc_shiftmax_t;

/* One integer ViT encoder block (LN -> QKV -> attention -> proj+res -> LN -> FC1+GELU -> FC2+res).
 * Weights are int8 row-major [out, in]; per-output-channel dyadic (mult, shift). */
typedef struct {
    int32_t d, H, F;          /* width, heads, MLP hidden */
    int32_t win_side;         /* 0 or 1: global attention; n: n x n windows on the token grid */
    int32_t ln_iters;         /* Newton iterations of I-LayerNorm */
    /* LN1 / LN2: per channel beta, signed multiplier, shift */
    const int32_t *ln1_beta, *ln1_mult, *ln1_shift;
    const int32_t *ln2_beta, *ln2_mult, *ln2_shift;
    /* QKV [3d, d] -> int8 q|k|v */
    const int8_t *w_qkv; const int32_t *b_qkv, *m_qkv, *s_qkv;
    /* attention */
    orc_shiftmax_t smx;
    int32_t m_o, s_o;         /* PV accumulator -> int8 O */
    /* proj [d, d] + residual -> int16 */
    const int8_t *w_proj; const int32_t *b_proj, *m_proj, *s_proj;
    int32_t m_r1, s_r1;       /* residual rescale of x */
    /* FC1 [F, d] -> int16 g -> SD-ShiftGELU -> int8 h */
    const int8_t *w_fc1; const int32_t *b_fc1, *m_fc1, *s_fc1;
    int32_t gelu_I0, gelu_k_inter, gelu_k_out;
    int32_t m_g, s_g;         /* GELU output (int32) -> int8 h */
    /* FC2 [d, F] + residual -> int16 */
    const int8_t *w_fc2; const int32_t *b_fc2, *m_fc2, *s_fc2;
    int32_t m_r2, s_r2;       /* residual rescale of x1 */
} orc_block_t;

/* Optional intermediate outputs of orc_block_forward (any pointer may be NULL). */
typedef struct {
    int8_t  *a1;   /* LN1 out      [B*T, d]  */
    int8_t  *qkv;  /* QKV out      [B*T, 3d] */
    int8_t  *o;    /* attention    [B*T, d]  */
    int16_t *x1;   /* after proj   [B*T, d]  */
    int8_t  *a2;   /* LN2 out      [B*T, d]  */
    int16_t *g;    /* FC1 out      [B*T, F]  */
    int8_t  *h;    /* GELU out     [B*T, F]  */
} orc_block_taps_t;

/* ---- scalar building blocks (exposed so the tests can pin them one by one) ---- */
int64_t orc_rq(int64_t v, int32_t m, int32_t s);
int64_t orc_sat(int64_t v, int32_t bits);
int64_t orc_shiftexp(int64_t I, int64_t I0, int32_t k_inter);          /* Algorithm 1 */
int32_t orc_calibrate_shift(int64_t S_sum, int32_t m_p, int32_t M_hw);  /* Algorithm 2 */
int64_t orc_sdshiftgelu_idiv(int64_t x, int32_t I0, int32_t k_inter, int32_t k_out);
int64_t orc_newton_isqrt(int64_t V, int32_t iters);

/* ---- tensor operators ---- */
void orc_shiftexp_vec(const int32_t *I, int64_t n, int32_t I0, int32_t k_inter, int64_t *out);

int orc_shiftmax_rows(const int32_t *X, int64_t ldx, int64_t rows, int64_t len,
                      const orc_shiftmax_t *p, uint8_t *P, int64_t ldp,
                      int64_t *S_sum_out /* rows, nullable */, int32_t *s_d_out /* rows, nullable */,
                      int64_t *S_R_out /* rows, nullable */);

int orc_sdshiftgelu(const int32_t *X, int32_t *Y, int64_t n, int32_t I0, int32_t k_inter,
                    int32_t k_out);

int orc_int_layernorm(const int32_t *X, int64_t ldx, int64_t rows, int64_t C,
                      const int32_t *beta, const int32_t *mult, const int32_t *shift,
                      int32_t iters, int32_t out_bits, int32_t *Y, int64_t ldy);

/* acc = A[M,K] . W[N,K]^T + bias (int64, must fit int32);
 * out_bits 8/16: sat(rq(acc; mult[c], shift[c]) [+ rq(res[row % res_rows, c]; m_r, s_r)]);
 * out_bits 32: acc itself (no requant, no residual). */
int orc_gemm_requant(const int8_t *A, int64_t lda, const int8_t *W, int64_t ldw,
                     const int32_t *bias, const int32_t *mult, const int32_t *shift,
                     int64_t M, int64_t N, int64_t K, int32_t out_bits,
                     const int16_t *res, int64_t ldr, int64_t res_rows, int32_t m_r, int32_t s_r,
                     int32_t *C, int64_t ldc);

/* Patch embedding: a p x p, stride-p integer convolution of the int8 image (NCHW), bias and
 * per-channel requantisation, plus the requantised position term, saturated to 16 bits:
 *   x0[b*T + t, c] = sat16(rq(acc; mult[c], shift[c]) + rq(pos[t, c]; m_pos, s_pos)),
 *   acc = bias[c] + sum_{ch,ky,kx} W[c, ch*p*p + ky*p + kx] * img[b, ch, py*p + ky, px*p + kx],
 * t = py * (Ww/p) + px.  pos may be NULL. */
int orc_patch_embed(const int8_t *img, int32_t B, int32_t Cin, int32_t Hh, int32_t Ww, int32_t p,
                    const int8_t *W, const int32_t *bias, const int32_t *mult, const int32_t *shift,
                    int32_t d, const int16_t *pos, int32_t m_pos, int32_t s_pos, int16_t *x0);

/* Multi-head attention on token-major q, k, v ([B*T, ld], head h at columns h*dh..h*dh+dh-1). */
int orc_attention(const int8_t *Q, const int8_t *K, const int8_t *V, int64_t ld,
                  int32_t B, int32_t T, int32_t H, int32_t dh, int32_t win_side,
                  const orc_shiftmax_t *p, int32_t m_o, int32_t s_o, int8_t *O, int64_t ldo);

int orc_block_forward(const orc_block_t *p, const int16_t *x, int16_t *y, int32_t B, int32_t T,
                      orc_block_taps_t *taps);

/* Scale-preserving split convolution (Sec. 3.2.2), 1x1 conv = per-pixel GEMM:
 * y[i,c] = sat8(rq( sum_b rq(X_b[i,:] . W_b[c,:]; m_b[b], s_b[b]) + bias[c]; mult[c], shift[c] )) */
int orc_split_conv(const int8_t *const *X, const int64_t *ldx, int32_t nb, int64_t M,
                   const int32_t *Kb, const int8_t *const *W, const int32_t *m_b,
                   const int32_t *s_b, const int32_t *bias, const int32_t *mult,
                   const int32_t *shift, int64_t N, int8_t *Y, int64_t ldy);

/* Integer deformable-attention sampling with nearest-neighbour lookup (Sec. 3.1.1). */
int orc_deform_attn(const int8_t *value, const int32_t *level_hw /* [L,2] (H_l, W_l) */,
                    int32_t L, const int32_t *ref_q16 /* [B,Q,2] (x,y) */,
                    const int32_t *off_q8 /* [B,Q,H,L,P,2] */, const uint8_t *w /* [B,Q,H,L*P] */,
                    int32_t B, int32_t Q, int32_t H, int32_t P, int32_t dh, int64_t S_total,
                    int32_t m, int32_t s, int8_t *out /* [B,Q,H*dh] */);

/* Per-tensor requantisation with an optional second term:
 *   Y[r,c] = sat_{out_bits}( rq(X[r,c]; m1, s1) + rq(Z[r mod z_rows, c]; m2, s2) ), Z may be NULL;
 * out_bits 8 / 16 saturate, 32 must fit int32. */
int orc_requant(const int32_t *X, int64_t ldx, int64_t rows, int64_t C, int32_t m1, int32_t s1,
                const int32_t *Z, int64_t ldz, int64_t z_rows, int32_t m2, int32_t s2,
                int32_t out_bits, int32_t *Y, int64_t ldy);

/* Nearest-neighbour resampling of B maps [Hi, Wi, C] to [Ho, Wo, C] (batch strides in rows):
 * Y[b][y*Wo + x] = X[b][floor(y*Hi/Ho)*Wi + floor(x*Wi/Wo)]. */
int orc_resample_nearest(const int8_t *X, int64_t x_bstride, int32_t B, int32_t Hi, int32_t Wi,
                         int32_t C, int8_t *Y, int64_t y_bstride, int32_t Ho, int32_t Wo);

/* Integer sigmoid of the detection head (Table 5: the head's exponential is ShiftExp), in the
 * sign-dependent form of SD-ShiftGELU's sigmoid factor (Sec. 3.3.1, Algorithm 1) with the logit
 * itself as the argument: out = (E F) >> (32 - k_out), scale 2^-(k_out-1). */
int64_t orc_int_sigmoid1(int64_t x, int32_t I0, int32_t k_inter, int32_t k_out);
int orc_int_sigmoid(const int32_t *X, int32_t *Y, int64_t n, int32_t I0, int32_t k_inter,
                    int32_t k_out);

/* Integer top-K (two-stage query selection): per row r of S [rows, lds], the K largest of its
 * first N values in decreasing order, equal values by increasing index. */
int orc_topk(const int32_t *S, int64_t lds, int32_t rows, int32_t N, int32_t K, int32_t *vals,
             int32_t *idx);

/* Row gather: dst row i = src row idx[i] (row_bytes bytes each; strides in bytes). */
int orc_gather_rows(const uint8_t *src, int64_t src_ld, int64_t src_rows, const int32_t *idx,
                    int64_t n, int64_t row_bytes, uint8_t *dst, int64_t dst_ld);

/* I-ViT's ShiftGELU (the ablation baseline of Sec. 3.3.1): per row, the sigmoid's exponentials are
 * taken after subtracting the row maximum of 1.702 x (clamped at 0, a reading):
 *   I_p = 1.702 I_x (shifts); M = max(max_row I_p, 0); E = ShiftExp(I_p - M); E' = ShiftExp(-M);
 *   I_div = (E * floor((2^31 - 1) / (E + E'))) >> (32 - k_out); Y = I_x * I_div. */
int orc_ivit_shiftgelu(const int32_t *X, int64_t ldx, int64_t rows, int64_t L, int32_t I0,
                       int32_t k_inter, int32_t k_out, int32_t *Y, int64_t ldy);

#ifdef __cplusplus
}
#endif
#endif
