// ilw_oracle.cpp -- plain, slow CPU oracle of the integer-only I-LW-DETR forward path.
//
// TEST INFRASTRUCTURE ONLY: used by tests/, __graft_entry__.smoke() and bench.py's CPU
// baseline.  It shares no code with the CUDA path.  Every loop is the textbook loop; nothing
// is blocked, fused or reordered beyond what the cited definition states.
//
// Parity status per function (how each is pinned is listed in tests/test_oracle_pins.py):
//   orc_rq, orc_sat, orc_shiftexp, orc_calibrate_shift, orc_shiftmax_rows,
//   orc_sdshiftgelu(_idiv), orc_newton_isqrt, orc_int_layernorm, orc_gemm_requant,
//   orc_attention, orc_split_conv, orc_deform_attn, orc_patch_embed, orc_requant,
//   orc_resample_nearest, orc_int_sigmoid, orc_topk, orc_gather_rows, orc_ivit_shiftgelu : pinned.
//   orc_block_forward : its structure (a pre-norm block, two-term residual requantisation, windows
//   cut from the row-major token grid) is a reading; pinned by reductions and invariants: with
//   constant branches it is two residual adds, with uniform scores its attention is a closed
//   form, with a constant hidden layer its MLP is one SD-ShiftGELU value per column, a per-token
//   offset passes through it, windowed equals global per window, tokens are equivariant.
// Each operator is written from its mathematics as the cited passage defines it; where the paper
// proves two forms equal (Constrained Shiftmax's reduced denominator), the plain form is used and
// a pin checks the other.
#include "ilw_oracle.h"

#include <cstdint>
#include <cstdlib>
#include <algorithm>
#include <vector>

namespace {

constexpr int64_t kInt31Max = (int64_t(1) << 31) - 1;  // 2^31 - 1

// floor(a / b) for any signs, b != 0.
int64_t floor_div(int64_t a, int64_t b) {
    int64_t q = a / b;
    if ((a % b != 0) && ((a < 0) != (b < 0))) q -= 1;
    return q;
}

int64_t clamp64(int64_t v, int64_t lo, int64_t hi) { return v < lo ? lo : (v > hi ? hi : v); }

// The fixed-point quotient shared by Constrained Shiftmax's normalisation (Sec. 3.3.2) and, with
// s_d = 0, by IntDiv (a reading): num / den with k_out - 1 fractional bits, formed as a 31-bit
// reciprocal F = floor((2^31 - 1) / den') of the denominator den' = clamp(den >> s_d, 1, 2^31 - 1)
// and a right shift of num F by 31 - (k_out - 1) + s_d.  `den_reduced` is den >> s_d.
int64_t fixed_point_ratio(int64_t num, int64_t den_reduced, int32_t s_d, int32_t k_out) {
    const int64_t F = kInt31Max / clamp64(den_reduced, 1, kInt31Max);
    return (int64_t)(((__int128)num * F) >> (31 - (k_out - 1) + s_d));
}

}  // namespace

extern "C" {

// Dyadic requantisation (Sec. 3.2.2: a fixed rescale applied as an integer multiply followed by a
// right shift).  Reading: round half up, i.e. add 2^(s-1) before the arithmetic right shift.  Computed in int128 so that no
// intermediate can overflow; the callers' ranges keep the result within int64.
int64_t orc_rq(int64_t v, int32_t m, int32_t s) {
    __int128 p = (__int128)v * (__int128)m;
    if (s <= 0) return (int64_t)p;
    p += (__int128)1 << (s - 1);
    return (int64_t)(p >> s);
}

// Symmetric saturation to N bits (Sec. 3.2.1: symmetric quantisation, no zero-point).
int64_t orc_sat(int64_t v, int32_t bits) {
    int64_t hi = (int64_t(1) << (bits - 1)) - 1;
    return clamp64(v, -hi, hi);
}

// ShiftExp (Algorithm 1, Sec. 3.3.1): an integer stand-in for e^(S I), I <= 0, where the caller
// supplies I0 = round(1/S) instead of S.  Since e^(S I) = 2^(S I log2 e), the input is first
// brought to base 2 with shifts and adds, I_e = I + floor(I/2) - floor(I/16) (log2 e ~ 1.4375,
// each shift flooring as an arithmetic shift does).  Its magnitude t = -I_e, in units of 1/I0, is
// clipped at k_inter I0 (powers below 2^-k_inter are all represented by the smallest one) and
// divided with remainder, t = q I0 + r, 0 <= r < I0: 2^(-t/I0) = 2^-q 2^(-r/I0).  The fractional
// power is replaced by its chord 2^-f ~ 1 - f/2 on [0, 1), so I0 2^(-r/I0) becomes I0 - r/2, rounded
// the way Algorithm 1 rounds it (a floor of -r/2, i.e. I0 - ceil(r/2)).  The integer power 2^-q and
// k_inter fractional bits of output scale (S_exp = S / 2^k_inter) leave one left shift by k_inter - q.
int64_t orc_shiftexp(int64_t I, int64_t I0, int32_t k_inter) {
    const int64_t I_e = I + floor_div(I, 2) - floor_div(I, 16);  // I log2 e
    const int64_t t = std::min(-I_e, (int64_t)k_inter * I0);     // clipped magnitude of the exponent
    const int64_t q = t / I0, r = t % I0;                         // t = q I0 + r (t >= 0)
    const int64_t I_b = I0 - (r + 1) / 2;                         // I0 2^(-r/I0) by the chord
    return I_b << (k_inter - q);
}

// CalibrateShift (Algorithm 2, Sec. 3.3.2): the smallest denominator shift s_d >= 0 that leaves a
// sum of ceil(log2 S_sum) bits with m_p bits of headroom below the M_hw-bit division:
// s_d = max(ceil(log2 S_sum) + m_p - M_hw, 0), where ceil(log2 S) is the least m with 2^m >= S.
int32_t orc_calibrate_shift(int64_t S_sum, int32_t m_p, int32_t M_hw) {
    int32_t bits_needed = 0;
    while (bits_needed < 62 && (int64_t(1) << bits_needed) < S_sum) ++bits_needed;
    return std::max(bits_needed + m_p - M_hw, 0);
}

void orc_shiftexp_vec(const int32_t *I, int64_t n, int32_t I0, int32_t k_inter, int64_t *out) {
    for (int64_t i = 0; i < n; ++i) out[i] = orc_shiftexp(I[i], I0, k_inter);
}

// Constrained Shiftmax (Algorithm 2, Sec. 3.3.2): softmax_i = e^(x_i - max) / sum_j e^(x_j - max)
// over each row, every exponential by ShiftExp (its argument x_i - max is never positive).  The
// exponentials are summed exactly (S_sum, int64).  The sum is reduced by 2^s_d -- s_d from
// CalibrateShift per row, or a fixed s_d >= 0 -- so that the 31-bit reciprocal keeps precision: the
// paper accumulates the reduced sum as quotients plus the floored sum of remainders and shows that
// this equals floor(S_sum / 2^s_d), which is what is taken here.  The quotient is then the fixed-point
// ratio above with k_out - 1 fractional bits (outputs stored as u8: every one is < 2^k_out for
// k_out <= 8; a larger value is reported as error -3).
int orc_shiftmax_rows(const int32_t *X, int64_t ldx, int64_t rows, int64_t len,
                      const orc_shiftmax_t *p, uint8_t *P, int64_t ldp, int64_t *S_sum_out,
                      int32_t *s_d_out, int64_t *S_R_out) {
    if (p->I0 < 1 || p->k_inter < 0 || p->k_inter > 30 || p->k_out < 1 || p->k_out > 8)
        return -1;
    if (len < 0 || rows < 0) return -1;
    std::vector<int64_t> e((size_t)len);
    for (int64_t row = 0; row < rows; ++row) {
        const int32_t *x = X + row * ldx;
        uint8_t *out = P + row * ldp;
        if (len == 0) {
            if (S_sum_out) S_sum_out[row] = 0;
            if (s_d_out) s_d_out[row] = 0;
            if (S_R_out) S_R_out[row] = 0;
            continue;
        }
        const int64_t x_max = *std::max_element(x, x + len);
        int64_t S_sum = 0;
        for (int64_t i = 0; i < len; ++i) {
            e[i] = orc_shiftexp((int64_t)x[i] - x_max, p->I0, p->k_inter);
            S_sum += e[i];
        }
        const int32_t s_d = p->s_d >= 0 ? p->s_d : orc_calibrate_shift(S_sum, p->m_p, p->M_hw);
        const int64_t S_R = clamp64(S_sum >> s_d, 1, kInt31Max);
        for (int64_t i = 0; i < len; ++i) {
            const int64_t o = fixed_point_ratio(e[i], S_sum >> s_d, s_d, p->k_out);
            if (o < 0 || o > 255) return -3;
            out[i] = (uint8_t)o;
        }
        if (S_sum_out) S_sum_out[row] = S_sum;
        if (s_d_out) s_d_out[row] = s_d;
        if (S_R_out) S_R_out[row] = S_R;
    }
    return 0;
}

// SD-ShiftGELU (Algorithm 1, Sec. 3.3.1): GELU(x) ~ x sigma(1.702 x).  The sigmoid is evaluated in
// its sign-split form sigma(z) = e^min(z,0) / (e^min(z,0) + e^-max(z,0)), in which neither
// exponential sees a positive argument, so no row maximum is needed and each element stands alone.
// z = 1.702 x is formed with shifts, I_p = x + floor(x/2) + floor(x/8) + floor(x/16) (1.6875 x);
// both exponentials come from ShiftExp; the quotient (IntDiv, which the paper does not define) is
// read as the fixed-point ratio of Constrained Shiftmax with s_d = 0.  Returns the sigmoid factor
// I_div (scale 2^-(k_out-1)); the GELU output is x I_div.
int64_t orc_sdshiftgelu_idiv(int64_t x, int32_t I0, int32_t k_inter, int32_t k_out) {
    const int64_t I_p = x + floor_div(x, 2) + floor_div(x, 8) + floor_div(x, 16);
    const int64_t I_shift = std::max<int64_t>(I_p, 0);
    const int64_t e_neg = orc_shiftexp(I_p - I_shift, I0, k_inter);  // e^min(z, 0)
    const int64_t e_pos = orc_shiftexp(-I_shift, I0, k_inter);       // e^-max(z, 0)
    return fixed_point_ratio(e_neg, e_neg + e_pos, 0, k_out);
}

int orc_sdshiftgelu(const int32_t *X, int32_t *Y, int64_t n, int32_t I0, int32_t k_inter,
                    int32_t k_out) {
    if (I0 < 1 || k_inter < 0 || k_inter > 30 || k_out < 1 || k_out > 16) return -1;
    for (int64_t i = 0; i < n; ++i) {
        int64_t idiv = orc_sdshiftgelu_idiv(X[i], I0, k_inter, k_out);
        int64_t o = (int64_t)X[i] * idiv;
        if (o < INT32_MIN || o > INT32_MAX) return -2;
        Y[i] = (int32_t)o;
    }
    return 0;
}

// Integer square root by Newton's method as used by I-LayerNorm (Sec. 3.3: I-ViT's LayerNorm,
// 10 iterations in the encoder, 20 in the decoder).  Reading: start at 2^16, run exactly
// `iters` steps x <- floor((x + floor(V/x)) / 2), stop early only if x reaches 0 (V = 0),
// and return max(x, 1).
int64_t orc_newton_isqrt(int64_t V, int32_t iters) {
    int64_t x = int64_t(1) << 16;
    for (int32_t it = 0; it < iters; ++it) {
        if (x == 0) break;
        x = floor_div(x + floor_div(V, x), 2);
    }
    return x < 1 ? 1 : x;
}

// I-LayerNorm (Sec. 3.3, the I-ViT integer LayerNorm).  Reading of the steps the paper leaves
// implicit:
//   mu = floor((2*sum(x) + C) / (2C))   (mean rounded half up)
//   y  = x - mu;  V = sum(y^2)
//   R  = NewtonIsqrt(V, iters);  F = floor((2^31-1) / R)
//   n  = (y * F) >> 1                   (normalised value, scale sqrt(C) / 2^30)
//   out = sat_{out_bits}( rq(n + beta_c; mult_c, shift_c) )   (gamma's sign and size in mult_c)
int orc_int_layernorm(const int32_t *X, int64_t ldx, int64_t rows, int64_t C, const int32_t *beta,
                      const int32_t *mult, const int32_t *shift, int32_t iters, int32_t out_bits,
                      int32_t *Y, int64_t ldy) {
    if (C < 1 || iters < 0 || (out_bits != 8 && out_bits != 16)) return -1;
    std::vector<int64_t> yv((size_t)C);
    for (int64_t r = 0; r < rows; ++r) {
        const int32_t *x = X + r * ldx;
        int64_t sum = 0;
        for (int64_t c = 0; c < C; ++c) sum += x[c];
        int64_t mu = floor_div(2 * sum + C, 2 * C);
        int64_t V = 0;
        for (int64_t c = 0; c < C; ++c) {
            yv[c] = (int64_t)x[c] - mu;
            V += yv[c] * yv[c];
        }
        int64_t R = orc_newton_isqrt(V, iters);
        int64_t F = kInt31Max / R;
        for (int64_t c = 0; c < C; ++c) {
            int64_t n = (yv[c] * F) >> 1;
            Y[r * ldy + c] = (int32_t)orc_sat(orc_rq(n + beta[c], mult[c], shift[c]), out_bits);
        }
    }
    return 0;
}

// Integer linear layer (Sec. 3.2.1, Eq. for Y ~ S_x S_w (I_x I_w) + b): the MAC runs in the
// integer domain, the scale is applied after accumulation as a per-output-channel dyadic
// requantisation.  Reading for the residual form: a second term rq(res; m_r, s_r) brings the
// residual stream to the output scale before the 16-bit saturation.
int orc_gemm_requant(const int8_t *A, int64_t lda, const int8_t *W, int64_t ldw,
                     const int32_t *bias, const int32_t *mult, const int32_t *shift, int64_t M,
                     int64_t N, int64_t K, int32_t out_bits, const int16_t *res, int64_t ldr,
                     int64_t res_rows, int32_t m_r, int32_t s_r, int32_t *C, int64_t ldc) {
    if (out_bits != 8 && out_bits != 16 && out_bits != 32) return -1;
    for (int64_t i = 0; i < M; ++i) {
        for (int64_t c = 0; c < N; ++c) {
            int64_t acc = 0;
            for (int64_t k = 0; k < K; ++k) acc += (int64_t)A[i * lda + k] * (int64_t)W[c * ldw + k];
            if (bias) acc += bias[c];
            if (acc < INT32_MIN || acc > INT32_MAX) return -2;
            int64_t v;
            if (out_bits == 32) {
                v = acc;
            } else {
                v = orc_rq(acc, mult[c], shift[c]);
                if (res) v += orc_rq(res[(i % res_rows) * ldr + c], m_r, s_r);
                v = orc_sat(v, out_bits);
            }
            C[i * ldc + c] = (int32_t)v;
        }
    }
    return 0;
}

// Patch embedding of the ViT encoder (Table 1: 640x640 input, 16x16 patches -> 1600 tokens):
// an integer convolution with kernel = stride = p (Sec. 3.2.1: integer MAC, scale after
// accumulation; Table 10 maps it to CONV_2D), written as the direct convolution sum.  The
// position term is a second requantised addend (the same two-term form as the residuals).
int orc_patch_embed(const int8_t *img, int32_t B, int32_t Cin, int32_t Hh, int32_t Ww, int32_t p,
                    const int8_t *W, const int32_t *bias, const int32_t *mult, const int32_t *shift,
                    int32_t d, const int16_t *pos, int32_t m_pos, int32_t s_pos, int16_t *x0) {
    if (p < 1 || Hh % p || Ww % p) return -1;
    const int32_t Gh = Hh / p, Gw = Ww / p, T = Gh * Gw, Kc = Cin * p * p;
    for (int32_t b = 0; b < B; ++b) {
        for (int32_t py = 0; py < Gh; ++py) {
            for (int32_t px = 0; px < Gw; ++px) {
                const int32_t t = py * Gw + px;
                for (int32_t c = 0; c < d; ++c) {
                    int64_t acc = bias ? bias[c] : 0;
                    for (int32_t ch = 0; ch < Cin; ++ch)
                        for (int32_t ky = 0; ky < p; ++ky)
                            for (int32_t kx = 0; kx < p; ++kx)
                                acc += (int64_t)W[(int64_t)c * Kc + (ch * p + ky) * p + kx] *
                                       img[(((int64_t)b * Cin + ch) * Hh + py * p + ky) * Ww + px * p + kx];
                    if (acc < INT32_MIN || acc > INT32_MAX) return -2;
                    int64_t v = orc_rq(acc, mult[c], shift[c]);
                    if (pos) v += orc_rq(pos[(int64_t)t * d + c], m_pos, s_pos);
                    x0[((int64_t)b * T + t) * d + c] = (int16_t)orc_sat(v, 16);
                }
            }
        }
    }
    return 0;
}

// Multi-head attention with Constrained Shiftmax.  Scores are the integer q.k^T (the 1/sqrt(dh)
// factor lives in the score scale, hence in I0); P = ConstrainedShiftmax(scores) (u8, scale
// 2^-(k_out-1)); O = P.V accumulated in int64, O8 = sat8(rq(O; m_o, s_o)).
// Attention groups: win_side <= 1 -> all T tokens; win_side = n -> the sqrt(T) x sqrt(T) token
// grid (row-major) is cut into n x n windows, tokens attend within their window only.
int orc_attention(const int8_t *Q, const int8_t *K, const int8_t *V, int64_t ld, int32_t B,
                  int32_t T, int32_t H, int32_t dh, int32_t win_side, const orc_shiftmax_t *p,
                  int32_t m_o, int32_t s_o, int8_t *O, int64_t ldo) {
    int32_t nw = win_side <= 1 ? 1 : win_side;
    int32_t G = 0, ws = 0;
    if (nw > 1) {
        while ((int64_t)(G + 1) * (G + 1) <= T) ++G;
        if ((int64_t)G * G != T || G % nw != 0) return -1;
        ws = G / nw;
    }
    int32_t Tg = nw > 1 ? ws * ws : T;
    std::vector<int64_t> tok((size_t)Tg);
    std::vector<int32_t> scores((size_t)Tg * Tg);
    std::vector<uint8_t> Pm((size_t)Tg * Tg);
    for (int32_t b = 0; b < B; ++b) {
        for (int32_t wy = 0; wy < nw; ++wy) {
            for (int32_t wx = 0; wx < nw; ++wx) {
                // token indices of this group, in local row-major order
                for (int32_t t = 0; t < Tg; ++t) {
                    if (nw > 1) {
                        int32_t ly = t / ws, lx = t % ws;
                        tok[t] = (int64_t)b * T + (int64_t)(wy * ws + ly) * G + (wx * ws + lx);
                    } else {
                        tok[t] = (int64_t)b * T + t;
                    }
                }
                for (int32_t h = 0; h < H; ++h) {
                    for (int32_t i = 0; i < Tg; ++i) {
                        for (int32_t j = 0; j < Tg; ++j) {
                            int64_t s = 0;
                            for (int32_t e = 0; e < dh; ++e)
                                s += (int64_t)Q[tok[i] * ld + h * dh + e] * K[tok[j] * ld + h * dh + e];
                            scores[(size_t)i * Tg + j] = (int32_t)s;
                        }
                    }
                    int rc = orc_shiftmax_rows(scores.data(), Tg, Tg, Tg, p, Pm.data(), Tg, nullptr,
                                               nullptr, nullptr);
                    if (rc) return rc;
                    for (int32_t i = 0; i < Tg; ++i) {
                        for (int32_t e = 0; e < dh; ++e) {
                            int64_t acc = 0;
                            for (int32_t j = 0; j < Tg; ++j)
                                acc += (int64_t)Pm[(size_t)i * Tg + j] * V[tok[j] * ld + h * dh + e];
                            O[tok[i] * ldo + h * dh + e] = (int8_t)orc_sat(orc_rq(acc, m_o, s_o), 8);
                        }
                    }
                }
            }
        }
    }
    return 0;
}

// One integer encoder block, composed exactly in this order (a reading; the paper fixes the
// operators, LW-DETR's plain ViT block fixes the order):
//   a1 = LN1(x); qkv = Linear_qkv(a1) -> int8; O = Attention(q, k, v);
//   x1 = sat16(rq(Linear_proj(O)) + rq(x)); a2 = LN2(x1);
//   g  = sat16(rq(Linear_fc1(a2))); h = sat8(rq(g * SDShiftGELU_Idiv(g); m_g, s_g));
//   y  = sat16(rq(Linear_fc2(h)) + rq(x1)).
int orc_block_forward(const orc_block_t *p, const int16_t *x, int16_t *y, int32_t B, int32_t T,
                      orc_block_taps_t *taps) {
    const int64_t Mt = (int64_t)B * T;
    const int32_t d = p->d, F = p->F;
    std::vector<int32_t> x32((size_t)Mt * d), t32((size_t)Mt * 3 * d), f32((size_t)Mt * F);
    std::vector<int8_t> a1((size_t)Mt * d), qkv((size_t)Mt * 3 * d), o((size_t)Mt * d);
    std::vector<int8_t> a2((size_t)Mt * d), h((size_t)Mt * F);
    std::vector<int16_t> x1((size_t)Mt * d), g((size_t)Mt * F);
    int rc;
    for (int64_t i = 0; i < Mt * d; ++i) x32[i] = x[i];
    rc = orc_int_layernorm(x32.data(), d, Mt, d, p->ln1_beta, p->ln1_mult, p->ln1_shift,
                           p->ln_iters, 8, t32.data(), d);
    if (rc) return rc;
    for (int64_t i = 0; i < Mt * d; ++i) a1[i] = (int8_t)t32[i];
    rc = orc_gemm_requant(a1.data(), d, p->w_qkv, d, p->b_qkv, p->m_qkv, p->s_qkv, Mt, 3 * d, d, 8,
                          nullptr, 0, 1, 0, 0, t32.data(), 3 * d);
    if (rc) return rc;
    for (int64_t i = 0; i < Mt * 3 * d; ++i) qkv[i] = (int8_t)t32[i];
    const int32_t dh = d / p->H;
    rc = orc_attention(qkv.data(), qkv.data() + d, qkv.data() + 2 * d, 3 * d, B, T, p->H, dh,
                       p->win_side, &p->smx, p->m_o, p->s_o, o.data(), d);
    if (rc) return rc;
    rc = orc_gemm_requant(o.data(), d, p->w_proj, d, p->b_proj, p->m_proj, p->s_proj, Mt, d, d, 16,
                          x, d, Mt, p->m_r1, p->s_r1, t32.data(), d);
    if (rc) return rc;
    for (int64_t i = 0; i < Mt * d; ++i) {
        x1[i] = (int16_t)t32[i];
        x32[i] = t32[i];
    }
    rc = orc_int_layernorm(x32.data(), d, Mt, d, p->ln2_beta, p->ln2_mult, p->ln2_shift,
                           p->ln_iters, 8, t32.data(), d);
    if (rc) return rc;
    for (int64_t i = 0; i < Mt * d; ++i) a2[i] = (int8_t)t32[i];
    rc = orc_gemm_requant(a2.data(), d, p->w_fc1, d, p->b_fc1, p->m_fc1, p->s_fc1, Mt, F, d, 16,
                          nullptr, 0, 1, 0, 0, f32.data(), F);
    if (rc) return rc;
    for (int64_t i = 0; i < Mt * F; ++i) {
        g[i] = (int16_t)f32[i];
        int64_t idiv = orc_sdshiftgelu_idiv(g[i], p->gelu_I0, p->gelu_k_inter, p->gelu_k_out);
        int64_t out = (int64_t)g[i] * idiv;
        h[i] = (int8_t)orc_sat(orc_rq(out, p->m_g, p->s_g), 8);
    }
    rc = orc_gemm_requant(h.data(), F, p->w_fc2, F, p->b_fc2, p->m_fc2, p->s_fc2, Mt, d, F, 16,
                          x1.data(), d, Mt, p->m_r2, p->s_r2, t32.data(), d);
    if (rc) return rc;
    for (int64_t i = 0; i < Mt * d; ++i) y[i] = (int16_t)t32[i];
    if (taps) {
        for (int64_t i = 0; i < Mt * d; ++i) {
            if (taps->a1) taps->a1[i] = a1[i];
            if (taps->o) taps->o[i] = o[i];
            if (taps->x1) taps->x1[i] = x1[i];
            if (taps->a2) taps->a2[i] = a2[i];
        }
        for (int64_t i = 0; i < Mt * 3 * d; ++i)
            if (taps->qkv) taps->qkv[i] = qkv[i];
        for (int64_t i = 0; i < Mt * F; ++i) {
            if (taps->g) taps->g[i] = g[i];
            if (taps->h) taps->h[i] = h[i];
        }
    }
    return 0;
}

// Scale-preserving split convolution (Sec. 3.2.2, Fig. 2(b)): each branch b is convolved with
// its own activation scale; its integer partial output is rescaled to the common scale (the
// maximum calibrated branch scale) by a dyadic multiply-and-shift (m_b, s_b); the rescaled
// partials are summed in the integer domain, the bias is added, and the per-output-channel
// requantisation gives the int8 output.  A 1x1 convolution is a per-pixel GEMM.
int orc_split_conv(const int8_t *const *X, const int64_t *ldx, int32_t nb, int64_t M,
                   const int32_t *Kb, const int8_t *const *W, const int32_t *m_b,
                   const int32_t *s_b, const int32_t *bias, const int32_t *mult,
                   const int32_t *shift, int64_t N, int8_t *Y, int64_t ldy) {
    if (nb < 1) return -1;
    for (int64_t i = 0; i < M; ++i) {
        for (int64_t c = 0; c < N; ++c) {
            int64_t total = 0;
            for (int32_t b = 0; b < nb; ++b) {
                int64_t acc = 0;
                for (int32_t k = 0; k < Kb[b]; ++k)
                    acc += (int64_t)X[b][i * ldx[b] + k] * (int64_t)W[b][c * Kb[b] + k];
                if (acc < INT32_MIN || acc > INT32_MAX) return -2;
                total += orc_rq(acc, m_b[b], s_b[b]);
            }
            total += bias ? bias[c] : 0;
            Y[i * ldy + c] = (int8_t)orc_sat(orc_rq(total, mult[c], shift[c]), 8);
        }
    }
    return 0;
}

// Integer deformable attention sampling (Sec. 3.1.1): bilinear interpolation replaced by the
// nearest grid point.  Reading: reference points are Q16 fractions of the feature map, offsets
// are Q8 pixels; the sample location in pixels is loc = ref * W_l + off, and the nearest grid
// point in the align_corners=False convention is floor(loc) (pixel centres at i + 1/2).
// Samples outside the map contribute 0.  The attention weights w are the Shiftmax outputs over
// the L*P samples of each (query, head); the weighted sum is requantised to int8.
int orc_deform_attn(const int8_t *value, const int32_t *level_hw, int32_t L,
                    const int32_t *ref_q16, const int32_t *off_q8, const uint8_t *w, int32_t B,
                    int32_t Q, int32_t H, int32_t P, int32_t dh, int64_t S_total, int32_t m,
                    int32_t s, int8_t *out) {
    std::vector<int64_t> start((size_t)L);
    int64_t acc_s = 0;
    for (int32_t l = 0; l < L; ++l) {
        start[l] = acc_s;
        acc_s += (int64_t)level_hw[2 * l] * level_hw[2 * l + 1];
    }
    if (acc_s != S_total) return -1;
    const int64_t Dm = (int64_t)H * dh;
    std::vector<int64_t> acc((size_t)dh);
    for (int32_t b = 0; b < B; ++b) {
        for (int32_t q = 0; q < Q; ++q) {
            int64_t rx = ref_q16[((int64_t)b * Q + q) * 2 + 0];
            int64_t ry = ref_q16[((int64_t)b * Q + q) * 2 + 1];
            for (int32_t h = 0; h < H; ++h) {
                for (int32_t e = 0; e < dh; ++e) acc[e] = 0;
                for (int32_t l = 0; l < L; ++l) {
                    int64_t Hl = level_hw[2 * l], Wl = level_hw[2 * l + 1];
                    for (int32_t pt = 0; pt < P; ++pt) {
                        int64_t base = ((((int64_t)b * Q + q) * H + h) * L + l) * P + pt;
                        int64_t ox = off_q8[base * 2 + 0], oy = off_q8[base * 2 + 1];
                        int64_t wt = w[(((int64_t)b * Q + q) * H + h) * (L * P) + l * P + pt];
                        int64_t px = ((rx * Wl) >> 8) + ox;  // Q8 pixels
                        int64_t py = ((ry * Hl) >> 8) + oy;
                        int64_t ix = px >> 8, iy = py >> 8;  // floor
                        if (ix < 0 || ix >= Wl || iy < 0 || iy >= Hl) continue;
                        const int8_t *v = value + ((int64_t)b * S_total + start[l] + iy * Wl + ix) * Dm + h * dh;
                        for (int32_t e = 0; e < dh; ++e) acc[e] += wt * v[e];
                    }
                }
                for (int32_t e = 0; e < dh; ++e)
                    out[((int64_t)b * Q + q) * Dm + h * dh + e] = (int8_t)orc_sat(orc_rq(acc[e], m, s), 8);
            }
        }
    }
    return 0;
}

// Per-tensor requantisation of an activation (the QuantAct that brings the int16 residual
// stream to the int8 input of the next integer linear layer, Sec. 3.2.1), with an optional
// second requantised term added before saturation (two tensors brought to one activation
// scale, as for the decoder's query plus positional query):
//   Y[r, c] = sat_{out_bits}( rq(X[r, c]; m1, s1) + rq(Z[r mod z_rows, c]; m2, s2) ),  Z may be NULL.
// out_bits 8 / 16 saturate symmetrically; out_bits 32 requires the sum to fit int32.
int orc_requant(const int32_t *X, int64_t ldx, int64_t rows, int64_t C, int32_t m1, int32_t s1,
                const int32_t *Z, int64_t ldz, int64_t z_rows, int32_t m2, int32_t s2,
                int32_t out_bits, int32_t *Y, int64_t ldy) {
    if (out_bits != 8 && out_bits != 16 && out_bits != 32) return -1;
    if (Z && z_rows < 1) return -1;
    for (int64_t r = 0; r < rows; ++r) {
        for (int64_t c = 0; c < C; ++c) {
            int64_t v = orc_rq(X[r * ldx + c], m1, s1);
            if (Z) v += orc_rq(Z[(r % z_rows) * ldz + c], m2, s2);
            if (out_bits == 32) {
                if (v < INT32_MIN || v > INT32_MAX) return -2;
                Y[r * ldy + c] = (int32_t)v;
            } else {
                Y[r * ldy + c] = (int32_t)orc_sat(v, out_bits);
            }
        }
    }
    return 0;
}

// Nearest-neighbour resampling of B feature maps (reading of the multi-scale projector's
// strides): map b of X is [Hi, Wi] pixels of C int8 channels, pixel (y, x) at row y*Wi + x of
// X + b*x_bstride rows; Y[b][y*Wo + x] = X[b][floor(y*Hi/Ho)*Wi + floor(x*Wi/Wo)].
int orc_resample_nearest(const int8_t *X, int64_t x_bstride, int32_t B, int32_t Hi, int32_t Wi,
                         int32_t C, int8_t *Y, int64_t y_bstride, int32_t Ho, int32_t Wo) {
    if (B < 0 || Hi < 1 || Wi < 1 || Ho < 1 || Wo < 1 || C < 1) return -1;
    for (int32_t b = 0; b < B; ++b)
        for (int32_t y = 0; y < Ho; ++y)
            for (int32_t x = 0; x < Wo; ++x) {
                const int64_t sy = (int64_t)y * Hi / Ho, sx = (int64_t)x * Wi / Wo;
                const int8_t *src = X + ((int64_t)b * x_bstride + sy * Wi + sx) * C;
                int8_t *dst = Y + ((int64_t)b * y_bstride + (int64_t)y * Wo + x) * C;
                for (int32_t c = 0; c < C; ++c) dst[c] = src[c];
            }
    return 0;
}

// Integer sigmoid of the detection head.  Table 5 lists ShiftExp as the integer form of the
// detection head's exponential; the sigmoid is taken in the sign-split form SD-ShiftGELU uses for
// its sigmoid factor (Sec. 3.3.1), sigma(z) = e^min(z,0) / (e^min(z,0) + e^-max(z,0)), with the logit
// itself as z (a reading: no 1.702 factor), and the same fixed-point quotient (k_out - 1 fractional
// bits).
int64_t orc_int_sigmoid1(int64_t x, int32_t I0, int32_t k_inter, int32_t k_out) {
    const int64_t x_pos = std::max<int64_t>(x, 0);
    const int64_t e_neg = orc_shiftexp(x - x_pos, I0, k_inter);  // e^min(z, 0)
    const int64_t e_pos = orc_shiftexp(-x_pos, I0, k_inter);     // e^-max(z, 0)
    return fixed_point_ratio(e_neg, e_neg + e_pos, 0, k_out);
}

int orc_int_sigmoid(const int32_t *X, int32_t *Y, int64_t n, int32_t I0, int32_t k_inter,
                    int32_t k_out) {
    if (I0 < 1 || k_inter < 0 || k_inter > 30 || k_out < 1 || k_out > 24) return -1;
    for (int64_t i = 0; i < n; ++i) Y[i] = (int32_t)orc_int_sigmoid1(X[i], I0, k_inter, k_out);
    return 0;
}

// Integer top-K of the two-stage query selection: the K largest values of each row,
// in decreasing order, equal values ordered by increasing index (a deterministic order the
// paper leaves open).  Plain selection: K times, the first index holding the largest value not
// yet taken.
int orc_topk(const int32_t *S, int64_t lds, int32_t rows, int32_t N, int32_t K, int32_t *vals,
             int32_t *idx) {
    if (rows < 0 || N < 1 || K < 1 || K > N) return -1;
    std::vector<char> taken((size_t)N);
    for (int32_t r = 0; r < rows; ++r) {
        const int32_t *s = S + (int64_t)r * lds;
        std::fill(taken.begin(), taken.end(), 0);
        for (int32_t k = 0; k < K; ++k) {
            int32_t best = -1;
            for (int32_t j = 0; j < N; ++j)
                if (!taken[(size_t)j] && (best < 0 || s[j] > s[best])) best = j;
            taken[(size_t)best] = 1;
            vals[(int64_t)r * K + k] = s[best];
            idx[(int64_t)r * K + k] = best;
        }
    }
    return 0;
}

int orc_gather_rows(const uint8_t *src, int64_t src_ld, int64_t src_rows, const int32_t *idx,
                    int64_t n, int64_t row_bytes, uint8_t *dst, int64_t dst_ld) {
    if (n < 0 || row_bytes < 0) return -1;
    for (int64_t i = 0; i < n; ++i) {
        if (idx[i] < 0 || idx[i] >= src_rows) return -1;
        for (int64_t b = 0; b < row_bytes; ++b) dst[i * dst_ld + b] = src[(int64_t)idx[i] * src_ld + b];
    }
    return 0;
}

// I-ViT's ShiftGELU, the baseline SD-ShiftGELU replaces (Sec. 3.3.1): the same sigmoid factor of
// 1.702 x, but with every exponential made non-positive by the row's maximum M of I_p instead of by
// each element's sign, sigma(z) = e^(z - M) / (e^(z - M) + e^-M).  A reading: M is clamped at 0 (a
// row whose values are all negative has M = 0, where the identity holds just the same and -M stays
// non-positive).
int orc_ivit_shiftgelu(const int32_t *X, int64_t ldx, int64_t rows, int64_t L, int32_t I0,
                       int32_t k_inter, int32_t k_out, int32_t *Y, int64_t ldy) {
    if (I0 < 1 || k_inter < 0 || k_inter > 30 || k_out < 1 || k_out > 16 || L < 1) return -1;
    std::vector<int64_t> Ip((size_t)L);
    for (int64_t r = 0; r < rows; ++r) {
        const int32_t *x = X + r * ldx;
        int64_t M = 0;
        for (int64_t c = 0; c < L; ++c) {
            const int64_t v = x[c];
            Ip[(size_t)c] = v + floor_div(v, 2) + floor_div(v, 8) + floor_div(v, 16);
            M = std::max(M, Ip[(size_t)c]);
        }
        const int64_t e_max = orc_shiftexp(-M, I0, k_inter);  // e^-M
        for (int64_t c = 0; c < L; ++c) {
            const int64_t e = orc_shiftexp(Ip[(size_t)c] - M, I0, k_inter);
            const int64_t o = (int64_t)x[c] * fixed_point_ratio(e, e + e_max, 0, k_out);
            if (o < INT32_MIN || o > INT32_MAX) return -2;
            Y[r * ldy + c] = (int32_t)o;
        }
    }
    return 0;
}

}  // extern "C"
