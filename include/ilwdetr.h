/*
 * ilwdetr.h -- C-ABI of the GB300 (sm_103a) integer-only I-LW-DETR forward path.
 *
 * Every entry point computes one integer operator of "Enabling Fully Integer-Only Inference for
 * Lightweight Detection Transformers" exactly (bit for bit) as the paper defines it; the
 * passages are cited beside each declaration.  All arithmetic on the device is integer.
 *
 * Conventions (apply to every call unless a declaration says otherwise)
 *   - Pointers to tensors are DEVICE pointers owned by the caller; the library never frees or
 *     keeps them.  Arrays described as "host" are read during the call only.
 *   - Layouts are row-major with an explicit leading dimension (elements between rows).
 *   - Every call is asynchronous on `stream` (0 = the legacy default stream) and returns an
 *     int status: ILW_OK, or a negative ILW_ERR_* code with a message available from
 *     ilwdetr_last_error() (thread-local).  Argument errors are reported before anything is
 *     launched.  Device-side failures that the kernels detect (a bounded wait that ran out)
 *     are latched in a device status word and reported by ilwdetr_device_status().
 *   - A call whose batch, row, token or element count is 0 checks its scalar parameters, returns
 *     ILW_OK and launches nothing; its tensor pointers may then be NULL.
 *   - rq(v; m, s) = (v*m + 2^(s-1)) >> s, arithmetic shift (dyadic requantisation, Sec. 3.2.2,
 *     round half up); satN clips to the symmetric range [-(2^(N-1)-1), 2^(N-1)-1] (Sec. 3.2.1).
 *     Per-channel `mult` is int32 (sign allowed), `shift` is int32 in [1, 62]; values outside
 *     that domain give unspecified results.
 *   - The caller passes integer parameters only (I0 = round(1/S), dyadic pairs, shifts): the
 *     float scales of calibration never reach the device.
 *   - The library keeps a few arrays of its own in device memory (the status word, the
 *     SD-ShiftGELU tables, the allocation-free patch scratch) and looks up their device
 *     addresses once per device.  A cudaDeviceReset ends the context those addresses belong
 *     to: do not call the library across one.  The SD-ShiftGELU GEMM epilogue keeps one 64 KB
 *     output table per distinct (I0, k_inter, k_out, m_g, s_g) for the life of the process, up
 *     to 256 per device; a GEMM with a further parameter set fails with ILW_ERR_CUDA (out of
 *     memory) and launches nothing.
 */
#ifndef ILWDETR_H
#define ILWDETR_H
#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *ilw_stream_t; /* identical to cudaStream_t */

enum {
    ILW_OK = 0,
    ILW_ERR_INVALID_ARG = -1, /* null / misaligned pointer, bad size, parameter out of domain */
    ILW_ERR_UNSUPPORTED = -2, /* valid but outside what the kernels implement (e.g. head dim) */
    ILW_ERR_CUDA = -3,        /* a CUDA runtime call or launch failed */
    ILW_ERR_TIMEOUT = -4      /* a kernel's bounded wait expired (see ilwdetr_device_status) */
};

/* Activation form code: int8-range integers (|v| <= 127) stored as fp16, which holds them exactly.
 * It is the operand form of the fp16 tensor-core kernels; a producer that writes it saves its
 * consumer the int8 -> fp16 conversion.  Accepted where an argument says so (out_bits of the
 * GEMMs and of ilwdetr_int_layernorm, a_form of ilwdetr_gemm, qkv_form and o_form of
 * ilwdetr_shiftmax_attn, a_form of ilwdetr_patch_embed's internal GEMM); 8 denotes plain int8. */
#define ILW_I8_IN_F16 108

/* Library version string, e.g. "ilwdetr 0.1 sm_103a". */
const char *ilwdetr_version(void);
/* Message of the last failing call on this thread ("" if none). */
const char *ilwdetr_last_error(void);
/* Synchronises `stream`, then reads and clears the device status word of the current device:
 * ILW_OK, ILW_ERR_TIMEOUT if a kernel gave up a bounded wait since the last read, or
 * ILW_ERR_INVALID_ARG if ilwdetr_gather_rows met an index outside its source since then. */
int ilwdetr_device_status(ilw_stream_t stream);

/* Constrained Shiftmax parameters (Algorithm 2 inputs; Sec. 3.3.2).
 *   I0      round(1/S_x) of the score scale, 1 <= I0 < 2^15 (ShiftExp, Algorithm 1)
 *   k_inter intermediate precision, 0 <= k_inter <= 16, I0 * 2^k_inter < 2^31
 *   k_out   output bits, 1 <= k_out <= 8 (outputs are u8 with scale 2^-(k_out-1))
 *   s_d     < 0: per-row CalibrateShift (Algorithm 2); >= 0: static shift (<= 31)
 *   m_p     precision margin (the paper uses 4); M_hw hardware division precision (31) */
typedef struct {
    int32_t I0, k_inter, k_out, s_d, m_p, M_hw;
} ilw_shiftmax_t;

/* SD-ShiftGELU parameters (Algorithm 1 inputs; Sec. 3.3.1).  1 <= I0, I0 * 2^(k_inter+1) < 2^31,
 * 1 <= k_out <= 8. */
typedef struct {
    int32_t I0, k_inter, k_out;
} ilw_gelu_t;

/* Residual term of a two-term requantised sum: out = sat(rq(acc) + rq(x[row % rows]; mult, shift)).
 * x is an int16 device tensor [rows, >= N] with leading dimension ldx. */
typedef struct {
    const int16_t *x;
    int64_t ldx;
    int64_t rows;
    int32_t mult, shift;
} ilw_residual_t;

/* ------------------------------------------------------------------ integer linear layers */

/* Bytes of the packed form of an int8 weight W[N, K] (row-major, K contiguous). */
size_t ilwdetr_packed_weight_bytes(int32_t N, int32_t K);
/* Packs W (device, int8 [N, K], leading dimension K) into `packed` (device, bytes given by
 * ilwdetr_packed_weight_bytes).  Done once per weight; the values stay the same integers (the
 * paper has no counterpart: this is the tensor cores' operand form of the int8 weights of
 * Sec. 3.2.1's integer linear layers).  K must be a multiple of 16. */
int ilwdetr_pack_weight(const int8_t *W, int32_t N, int32_t K, void *packed, ilw_stream_t stream);

/* Integer linear layer with fused bias and dyadic requantisation (Sec. 3.2.1, the equation
 * Y ~ S_x S_w (I_x I_w) + b: the MAC is integer, the scale is applied after accumulation).
 *   A      int8 [M, K] (lda >= K, lda and the base 16-byte aligned)
 *   Wp     packed weight of W int8 [N, K]
 *   acc[i,c] = sum_k A[i,k] W[c,k] + bias[c]      (exact; must fit int32)
 *   out_bits 8 / 16: C[i,c] = satN(rq(acc; mult[c], shift[c]) [+ rq(res...)]) (int8 / int16)
 *   out_bits 32    : C[i,c] = acc (int32; mult, shift and res ignored and may be NULL)
 *   out_bits ILW_I8_IN_F16: the out_bits 8 values, stored as fp16 (C is fp16 [M, ldc])
 *   bias may be NULL (0).  C has leading dimension ldc (elements).
 *   K: a multiple of 16.  Each output tile keeps one exact fp32 accumulator per 1024 terms of K in
 *   tensor memory, so K <= 2048 in every tile shape and K <= 4096 where 128-wide tiles are chosen;
 *   a K the chosen shape cannot hold is refused before any launch (ILW_ERR_CUDA, invalid argument). */
int ilwdetr_gemm_requant(const int8_t *A, int64_t lda, const void *Wp, const int32_t *bias,
                         const int32_t *mult, const int32_t *shift, int32_t M, int32_t N,
                         int32_t K, int32_t out_bits, void *C, int64_t ldc,
                         const ilw_residual_t *res /* nullable, host struct */,
                         ilw_stream_t stream);

/* Integer linear layer followed by SD-ShiftGELU (Sec. 3.3.1, Algorithm 1) in the epilogue:
 *   g = sat16(rq(acc; mult[c], shift[c]));  I_out = g * I_div(g)  (Algorithm 1, scale 2^-(k_out-1))
 *   H[i,c] = sat8(rq(I_out; m_g, s_g))  (int8, leading dimension ldh). */
int ilwdetr_gemm_gelu(const int8_t *A, int64_t lda, const void *Wp, const int32_t *bias,
                      const int32_t *mult, const int32_t *shift, int32_t M, int32_t N, int32_t K,
                      const ilw_gelu_t *gelu, int32_t m_g, int32_t s_g, int8_t *H, int64_t ldh,
                      ilw_stream_t stream);

/* The integer linear layer (Sec. 3.2.1) in its general form: the computation of ilwdetr_gemm_requant
 * (epilogue ILW_EPI_REQUANT) or of ilwdetr_gemm_gelu (ILW_EPI_GELU), with the activation operand
 * A either int8 (a_form 8; lda % 16 == 0) or the same int8 values carried in fp16 (a_form
 * ILW_I8_IN_F16; fp16 [M, lda], lda % 8 == 0), which the tensor cores read directly.  out_bits:
 * 8 / 16 / 32 / ILW_I8_IN_F16 for ILW_EPI_REQUANT, 8 or ILW_I8_IN_F16 for ILW_EPI_GELU (the int8
 * outputs carried in fp16).  res: residual term (ILW_EPI_REQUANT, out_bits != 32), or NULL;
 * gelu, m_g, s_g: ILW_EPI_GELU only.  struct_size = sizeof(ilw_gemm_t). */
#define ILW_EPI_REQUANT 0
#define ILW_EPI_GELU 1
typedef struct {
    uint32_t struct_size;
    const void *A;
    int32_t a_form;
    int64_t lda;
    const void *Wp;
    const int32_t *bias, *mult, *shift;
    int32_t M, N, K;
    int32_t epilogue;
    int32_t out_bits;
    void *C;
    int64_t ldc;
    const ilw_residual_t *res;
    const ilw_gelu_t *gelu;
    int32_t m_g, s_g;
} ilw_gemm_t;
int ilwdetr_gemm(const ilw_gemm_t *g, ilw_stream_t stream);

/* Scale-preserving split convolution (Sec. 3.2.2, Fig. 2(b)), 1x1 kernels (a per-pixel GEMM):
 *   y[i,c] = sat8(rq( sum_b rq(X_b[i,:] . W_b[c,:]; m_b[b], s_b[b]) + bias[c]; mult[c], shift[c] ))
 * Each branch keeps its own activation scale; (m_b, s_b) is the dyadic ratio S_b / max_b S_b
 * (must satisfy m_b <= 2^s_b).  X, ldx, Kb, Wp, m_b, s_b are HOST arrays of nb entries holding
 * device pointers / values; 1 <= nb <= 8, every K_b a multiple of 16. */
int ilwdetr_split_conv(const int8_t *const *X, const int64_t *ldx, int32_t nb, int32_t M,
                       const int32_t *Kb, const void *const *Wp, const int32_t *m_b,
                       const int32_t *s_b, const int32_t *bias, const int32_t *mult,
                       const int32_t *shift, int32_t N, int8_t *Y, int64_t ldy,
                       ilw_stream_t stream);

/* ------------------------------------------------------------------ nonlinear operators */

/* Constrained Shiftmax over rows (Algorithm 2; Sec. 3.3.2): X int32 [rows, len] (ldx) ->
 * P u8 [rows, len] (ldp), scale 2^-(k_out-1).  Per row: max, ShiftExp of the differences,
 * S_sum (int64), s_d, the exact shifted denominator S_R = floor(S_sum / 2^s_d) (quotient-
 * remainder accumulation), F = floor((2^31-1)/clamp(S_R,1,2^31-1)), out = (I_exp F) >> (32-k_out+s_d). */
int ilwdetr_shiftmax_rows(const int32_t *X, int64_t ldx, int64_t rows, int32_t len,
                          const ilw_shiftmax_t *p, uint8_t *P, int64_t ldp, ilw_stream_t stream);

/* SD-ShiftGELU (Algorithm 1; Sec. 3.3.1), element-wise: Y[i] = X[i] * I_div(X[i]) (int32, scale
 * S_x 2^-(k_out-1)); IntDiv is Algorithm 2's fixed-point division with s_d = 0.
 * Values must satisfy |X[i]| * 2^(k_out-1) < 2^31. */
int ilwdetr_sdshiftgelu(const int32_t *X, int32_t *Y, int64_t n, const ilw_gelu_t *p,
                        ilw_stream_t stream);

/* I-LayerNorm (Sec. 3.3: I-ViT's integer LayerNorm with a Newton integer square root; 10
 * iterations in the encoder, 20 in the decoder).  Per row of C values:
 *   mu = floor((2 sum x + C) / (2C)); y = x - mu; V = sum y^2; R = Newton(V) from 2^16, `iters`
 *   steps; F = floor((2^31-1)/max(R,1)); n = (y F) >> 1; out = sat_{out_bits}(rq(n + beta[c];
 *   mult[c], shift[c])).
 *   X: in_bits 16 (int16) or 32 (int32, |x| < 2^24), [rows, C] with leading dimension ldx.
 *   Y: out_bits 8 (int8) or 16 (int16), leading dimension ldy.  1 <= C <= 4096. */
int ilwdetr_int_layernorm(const void *X, int32_t in_bits, int64_t ldx, int64_t rows, int32_t C,
                          const int32_t *beta, const int32_t *mult, const int32_t *shift,
                          int32_t iters, void *Y, int32_t out_bits, int64_t ldy,
                          ilw_stream_t stream);

/* ------------------------------------------------------------------ attention */

/* Multi-head attention with Constrained Shiftmax (Sec. 3.2.1 integer MatMul, Sec. 3.3.2):
 *   scores = q k^T (int32; 1/sqrt(dh) is folded into the score scale, hence into p->I0),
 *   P = ConstrainedShiftmax(scores) (u8), O = P V (int32), out = sat8(rq(O; m_o, s_o)).
 * Q, K, V: token-major, element (b, t, h, e) at [(b*T + t) * ld_qkv + h*dh + e] (elements), in
 * the form qkv_form: 8 = int8, ILW_I8_IN_F16 = the same integers as fp16 (16-byte aligned rows;
 * q|k|v of one [B*T, 3*H*dh] buffer is the usual case).
 * O: element (b, t, h, e) at [(b*T + t) * ld_o + h*dh + e], in the form o_form (8 = int8,
 * ILW_I8_IN_F16 = the int8 values as fp16).
 * win_side <= 1: global attention over the T tokens; win_side = n >= 2: the sqrt(T) x sqrt(T)
 * token grid (row-major) is cut into n x n windows and tokens attend within their window
 * (LW-DETR's window attention, Table 1).  dh must be 32 or 64. */
int ilwdetr_shiftmax_attn(const void *Q, const void *K, const void *V, int64_t ld_qkv,
                          int32_t qkv_form, int32_t B, int32_t T, int32_t H, int32_t dh, int32_t win_side,
                          const ilw_shiftmax_t *p, int32_t m_o, int32_t s_o, void *O, int32_t o_form,
                          int64_t ld_o, ilw_stream_t stream);

/* Integer deformable-attention sampling with nearest-neighbour lookup (Sec. 3.1.1): for each
 * (b, q, h) and sample (l, p): loc = ((ref * W_l) >> 8) + off (Q8 pixels), index = loc >> 8
 * (the nearest grid point, pixel centres at i + 1/2); samples outside the map contribute 0;
 * acc = sum w * value (int32); out = sat8(rq(acc; m, s)).
 *   value   int8 [B, S_total, H*dh], levels concatenated row-major (S_total = sum H_l W_l)
 *   level_hw HOST int32 [L, 2] = (H_l, W_l); 1 <= L <= 8
 *   ref_q16 int32 [B, Q, 2] = (x, y) in [0, 2^16) of the map; off_q8 int32 [B, Q, H, L, P, 2]
 *   w       u8 [B, Q, H, L*P] (Shiftmax outputs over the L*P samples)
 *   out     int8 [B, Q, H*dh].  dh must be a multiple of 4. */
int ilwdetr_deform_attn(const int8_t *value, const int32_t *level_hw, int32_t L,
                        const int32_t *ref_q16, const int32_t *off_q8, const uint8_t *w,
                        int32_t B, int32_t Q, int32_t H, int32_t P, int32_t dh, int32_t m,
                        int32_t s, int8_t *out, ilw_stream_t stream);

/* ------------------------------------------------------------------ patch embedding */

/* Workspace bytes of ilwdetr_patch_embed (the gathered patch matrix, B*T x Cin*p*p int8). */
size_t ilwdetr_patch_embed_workspace_bytes(int32_t B, int32_t Cin, int32_t Hh, int32_t Ww, int32_t p);
/* ViT patch embedding: a p x p convolution with stride p of the int8 image (an integer linear
 * layer on each non-overlapping patch, Sec. 3.2.1; Table 10 maps it to CONV_2D):
 *   x0[b*T + t, c] = sat16(rq(acc; mult[c], shift[c]) + rq(pos[t, c]; m_pos, s_pos)),
 *   acc = bias[c] + sum_{ch,ky,kx} W[c, (ch*p + ky)*p + kx] img[b, ch, py*p + ky, px*p + kx],
 *   t = py*(Ww/p) + px, T = (Hh/p)(Ww/p).
 *   img  int8 [B, Cin, Hh, Ww] (NCHW, 16-byte aligned), Ww and p multiples of 16, p | Hh, p | Ww
 *   Wp   packed weight of W int8 [d, Cin*p*p];  pos int16 [T, d] or NULL
 *   x0   int16 [B*T, d];  workspace: >= ilwdetr_patch_embed_workspace_bytes, 256-byte aligned */
int ilwdetr_patch_embed(const int8_t *img, int32_t B, int32_t Cin, int32_t Hh, int32_t Ww, int32_t p,
                        const void *Wp, const int32_t *bias, const int32_t *mult, const int32_t *shift,
                        int32_t d, const int16_t *pos, int32_t m_pos, int32_t s_pos, int16_t *x0,
                        void *workspace, size_t workspace_bytes, ilw_stream_t stream);

/* Allocation-free patch embedding.  The paper has no counterpart: this entry point exists for
 * callers that cannot provide device memory to the library -- a host runtime that owns the
 * whole device-memory budget and forbids allocations inside its inference loop, or a
 * latency-critical loop that cannot afford cudaMalloc/cudaFree and their implicit
 * synchronisation.  It computes exactly what ilwdetr_patch_embed computes, with the same
 * arguments minus the workspace, and allocates nothing: the gathered patch matrix lives in a
 * fixed 8 MiB device array inside the library (ilwdetr_patch_embed_noalloc_max_bytes()),
 * which every GPU that loads the library holds until the process exits.
 *   - Batches needing more than that (B * (Hh/p) * (Ww/p) * Cin * p * p bytes; e.g. more than
 *     6 images of 3 x 640 x 640) are rejected with ILW_ERR_UNSUPPORTED and a message.
 *   - The first call on each device looks up the array's device address (cudaGetSymbolAddress)
 *     with that device current; make that first call before any stream capture.  The address is
 *     kept for the life of the process, so do not call this across a cudaDeviceReset.
 *   - Every argument is checked before anything is launched; errors as ilwdetr_patch_embed.
 *   - All calls share the one array and it keeps the last call's contents (each call overwrites
 *     every byte it reads, so nothing needs clearing).  Calls whose execution overlaps on the
 *     GPU (other streams, other threads) race on it: serialise them. */
size_t ilwdetr_patch_embed_noalloc_max_bytes(void);
int ilwdetr_patch_embed_noalloc(const int8_t *img, int32_t B, int32_t Cin, int32_t Hh, int32_t Ww,
                                int32_t p, const void *Wp, const int32_t *bias, const int32_t *mult,
                                const int32_t *shift, int32_t d, const int16_t *pos, int32_t m_pos,
                                int32_t s_pos, int16_t *x0, ilw_stream_t stream);

/* Argument validation without launching (the paper has no counterpart; off by default).  While
 * `on` is non-zero for the calling thread, every entry point that launches kernels (the operators,
 * the composite block, decoder-layer and patch-embedding calls, ilwdetr_patch_embed_noalloc and
 * ilwdetr_pack_weight) checks its arguments exactly as usual and then returns ILW_OK, or the error
 * it found, without any CUDA call that launches work or touches device memory.  Composite calls
 * check every step.  Lets a host runtime validate a whole schedule ahead of time, and works on a
 * machine without a device.  Call ilwdetr_validate_only(0) to launch again.  Always ILW_OK. */
int ilwdetr_validate_only(int32_t on);

/* Test hook of the bounded device waits (the paper has no counterpart; off by default).  Every
 * wait inside the kernels is bounded; when one runs out the kernel latches the device status word,
 * stops, drains the copies it issued, frees its tensor memory and returns, and
 * ilwdetr_device_status() then reports ILW_ERR_TIMEOUT.  This call makes that path testable
 * without a fault: GEMM launches made after it skip the operand load of their K-block counter
 * `skip_load` (so the wait for it never completes; -1 = none) and bound every wait by
 * `wait_cycles` SM clock cycles (0 = the default, about one second).  Process-wide; not for use
 * while other threads launch GEMMs.  Call ilwdetr_debug_gemm_wait(-1, 0) to restore. */
int ilwdetr_debug_gemm_wait(int32_t skip_load, int64_t wait_cycles);

/* ------------------------------------------------------------------ encoder block */

/* Integer parameters of one encoder block (all pointers are device pointers; weights packed
 * with ilwdetr_pack_weight).  The block computes (a reading of LW-DETR's plain ViT block with
 * the paper's integer operators):
 *   a1 = LN1(x) (int8); qkv = sat8(rq(a1 Wqkv^T + b)) (token-major q|k|v);
 *   O = Attention(q, k, v) (int8); x1 = sat16(rq(O Wproj^T + b) + rq(x; m_r1, s_r1));
 *   a2 = LN2(x1); g = sat16(rq(a2 W1^T + b)); h = sat8(rq(g * I_div(g); m_g, s_g));
 *   y = sat16(rq(h W2^T + b) + rq(x1; m_r2, s_r2)). */
typedef struct {
    uint32_t struct_size; /* sizeof(ilw_block_params_t) */
    int32_t d, H, F, win_side, ln_iters;
    const int32_t *ln1_beta, *ln1_mult, *ln1_shift;
    const int32_t *ln2_beta, *ln2_mult, *ln2_shift;
    const void *w_qkv; const int32_t *b_qkv, *m_qkv, *s_qkv;
    ilw_shiftmax_t smx;
    int32_t m_o, s_o;
    const void *w_proj; const int32_t *b_proj, *m_proj, *s_proj;
    int32_t m_r1, s_r1;
    const void *w_fc1; const int32_t *b_fc1, *m_fc1, *s_fc1;
    ilw_gelu_t gelu;
    int32_t m_g, s_g;
    const void *w_fc2; const int32_t *b_fc2, *m_fc2, *s_fc2;
    int32_t m_r2, s_r2;
} ilw_block_params_t;

/* Workspace bytes ilwdetr_block_forward needs for B*T tokens. */
size_t ilwdetr_block_workspace_bytes(int32_t B, int32_t T, int32_t d, int32_t F);
/* One encoder block (the ViT encoder of Sec. 3.1.1 with the integer operators of Sec. 3.2-3.3;
 * global or window attention as Table 1 assigns per layer): x int16 [B*T, d] -> y int16
 * [B*T, d] (x and y may not alias).
 * `workspace` is a device buffer of at least ilwdetr_block_workspace_bytes (256-byte aligned). */
int ilwdetr_block_forward(const ilw_block_params_t *p, const int16_t *x, int16_t *y, int32_t B,
                          int32_t T, void *workspace, size_t workspace_bytes, ilw_stream_t stream);

/* ------------------------------------------------------------------ detector: projector, decoder */

/* Per-tensor requantisation with an optional second term (the QuantAct between the int16 residual
 * stream and the int8 input of an integer linear layer, Sec. 3.2.1; with Z, two tensors brought to
 * one activation scale, as for a decoder query plus its positional query):
 *   Y[r, c] = sat_{out_bits}( rq(X[r, c]; m1, s1) + rq(Z[r mod z_rows, c]; m2, s2) )
 *   X  int16 (in_bits 16) or int32 (in_bits 32) [rows, ldx];  Z int16 [z_rows, ldz] or NULL
 *   Y  int8 / int16 (symmetric saturation) or int32 (out_bits 32: the sum must fit int32, no
 *      saturation) [rows, ldy].  C, ldx, ldz, ldy must be multiples of 4 and each base pointer
 *      aligned to 4 elements.
 * Shifts in [1, 62]; |X m1| and |Z m2| must stay below 2^62 (always so for int16 inputs);
 * errors as for the other entry points. */
int ilwdetr_requant(const void *X, int32_t in_bits, int64_t ldx, int64_t rows, int32_t C, int32_t m1,
                    int32_t s1, const int16_t *Z, int64_t ldz, int64_t z_rows, int32_t m2, int32_t s2,
                    int32_t out_bits, void *Y, int64_t ldy, ilw_stream_t stream);

/* Nearest-neighbour resampling of B int8 feature maps (the multi-scale projector of Sec. 3.2.2 and
 * Table 1: its strides 8 / 16 / 32 read as nearest resampling of the stride-16 encoder grid; a 1x1
 * convolution commutes with it):
 *   Y[b][y*Wo + x, :] = X[b][floor(y*Hi/Ho)*Wi + floor(x*Wi/Wo), :]
 *   X int8, map b starts at row b*x_bstride of C channels; Y likewise with y_bstride (so the
 *   levels can be written into one concatenated decoder memory).  C % 16 == 0, 16-byte aligned. */
int ilwdetr_resample_nearest(const int8_t *X, int64_t x_bstride, int32_t B, int32_t Hi, int32_t Wi,
                             int32_t C, int8_t *Y, int64_t y_bstride, int32_t Ho, int32_t Wo,
                             ilw_stream_t stream);

/* One integer decoder layer (post-norm, the Deformable-DETR order; the paper's decoder with
 * nearest-neighbour deformable sampling, Sec. 3.1.1, and I-LayerNorm with 20 Newton steps,
 * Sec. 3.3).  All weights are packed (ilwdetr_pack_weight) int8 [out, in]:
 *   self-attention   qk_in = sat8(rq(tgt; m_q1,s_q1) + rq(pos; m_q2,s_q2)), v_in = sat8(rq(tgt; m_v1,s_v1));
 *                    q|k = rq8(qk_in W_qk^T) [2d], v = rq8(v_in W_v^T) [d]; global attention over
 *                    the Q queries (dh = d / H); x1 = sat16(rq(O W_o^T) + rq(tgt; m_r1,s_r1));
 *                    t1 = LN1(x1) (int16)
 *   cross-attention  qc = sat8(rq(t1; m_c1,s_c1) + rq(pos; m_c2,s_c2)); value = rq8(memory W_val^T);
 *                    Q8 offsets = rq16(qc W_off^T) [H*L*P*2]; logits = rq16(qc W_att^T) [H*L*P];
 *                    weights = Constrained Shiftmax (smx_w) over each head's L*P logits;
 *                    s = ilwdetr_deform_attn(value, ..., m_s, s_s);
 *                    x2 = sat16(rq(s W_o2^T) + rq(t1; m_r2,s_r2)); t2 = LN2(x2)
 *   FFN              f = sat8(rq(t2; m_f,s_f)); h = GELU8(f W_fc1^T) [F];
 *                    x3 = sat16(rq(h W_fc2^T) + rq(t2; m_r3,s_r3)); out = LN3(x3) (int16) */
typedef struct ilw_decoder_params_t {
    uint32_t struct_size; /* sizeof(ilw_decoder_params_t) */
    int32_t d, H, F, L, P, ln_iters;
    int32_t m_q1, s_q1, m_q2, s_q2, m_v1, s_v1;
    const void *w_qk; const int32_t *b_qk, *m_qk, *s_qk;
    const void *w_v; const int32_t *b_v, *m_v, *s_v;
    ilw_shiftmax_t smx;
    int32_t m_o, s_o;
    const void *w_o; const int32_t *b_o, *m_oc, *s_oc;
    int32_t m_r1, s_r1;
    const int32_t *ln1_beta, *ln1_mult, *ln1_shift;
    int32_t m_c1, s_c1, m_c2, s_c2;
    const void *w_val; const int32_t *b_val, *m_val, *s_val;
    const void *w_off; const int32_t *b_off, *m_off, *s_off;
    const void *w_att; const int32_t *b_att, *m_att, *s_att;
    ilw_shiftmax_t smx_w;
    int32_t m_s, s_s;
    const void *w_o2; const int32_t *b_o2, *m_o2, *s_o2;
    int32_t m_r2, s_r2;
    const int32_t *ln2_beta, *ln2_mult, *ln2_shift;
    int32_t m_f, s_f;
    const void *w_fc1; const int32_t *b_fc1, *m_fc1, *s_fc1;
    ilw_gelu_t gelu;
    int32_t m_g, s_g;
    const void *w_fc2; const int32_t *b_fc2, *m_fc2, *s_fc2;
    int32_t m_r3, s_r3;
    const int32_t *ln3_beta, *ln3_mult, *ln3_shift;
} ilw_decoder_params_t;

/* Workspace bytes of ilwdetr_decoder_layer_forward for B*Q queries over B*S_total memory rows. */
size_t ilwdetr_decoder_workspace_bytes(int32_t B, int32_t Q, int64_t S_total, int32_t d, int32_t F,
                                       int32_t H, int32_t L, int32_t P);
/* tgt, pos int16 [B*Q, d]; memory int8 [B*S_total, d] (levels concatenated per image, as
 * ilwdetr_deform_attn reads them); level_hw HOST int32 [L, 2]; ref_q16 int32 [B, Q, 2];
 * out int16 [B*Q, d] (may not alias tgt).  d % 16 == 0, d / H in {32, 64}, F % 16 == 0.
 * workspace: >= ilwdetr_decoder_workspace_bytes, 256-byte aligned. */
int ilwdetr_decoder_layer_forward(const ilw_decoder_params_t *p, const int16_t *tgt, const int16_t *pos,
                                  const int8_t *memory, const int32_t *level_hw, int32_t L,
                                  const int32_t *ref_q16, int32_t B, int32_t Q, int16_t *out,
                                  void *workspace, size_t workspace_bytes, ilw_stream_t stream);

/* ------------------------------------------------------------------ detection head, two-stage selection */

/* Integer sigmoid parameters.  1 <= I0 < 2^15, 0 <= k_inter <= 16, I0 * 2^(k_inter+1) < 2^31,
 * 1 <= k_out <= 24. */
typedef struct {
    int32_t I0, k_inter, k_out;
} ilw_sigmoid_t;

/* Integer sigmoid of the detection head (Table 5: the head's exponential is ShiftExp), taken in
 * the sign-dependent form of SD-ShiftGELU's sigmoid factor (Sec. 3.3.1, Algorithm 1) with the logit
 * itself as the argument:
 *   I_shift = ReLU(x), I_delta = x - I_shift, E = ShiftExp(I_delta), E' = ShiftExp(-I_shift),
 *   Y = (E * floor((2^31 - 1) / (E + E'))) >> (32 - k_out)      (scale 2^-(k_out-1))
 * X, Y int32 [n] device (may alias), 16-byte aligned. */
int ilwdetr_int_sigmoid(const int32_t *X, int32_t *Y, int64_t n, const ilw_sigmoid_t *p, ilw_stream_t stream);

/* I-ViT's ShiftGELU, the baseline SD-ShiftGELU replaces (Sec. 3.3.1), over rows of L values: the
 * sigmoid's exponentials after subtracting the row maximum of 1.702 x (clamped at 0):
 *   I_p = x + (x >> 1) + (x >> 3) + (x >> 4); M = max(max_row I_p, 0);
 *   E = ShiftExp(I_p - M), E' = ShiftExp(-M), I_div = (E floor((2^31-1)/(E + E'))) >> (32 - k_out),
 *   Y = x I_div (int32; values must satisfy |x| 2^(k_out-1) < 2^31).
 * X [rows, ldx], Y [rows, ldy] int32 device, 4-byte aligned, ldx, ldy >= L >= 1. */
int ilwdetr_ivit_shiftgelu(const int32_t *X, int64_t ldx, int64_t rows, int32_t L, int32_t *Y, int64_t ldy,
                           const ilw_gelu_t *p, ilw_stream_t stream);

/* ReLU of int8 values (the hidden layers of the detection head's box branch, Table 5):
 * Y = max(X, 0).  X, Y device [n] (may alias), 4-byte aligned. */
int ilwdetr_relu_i8(const int8_t *X, int8_t *Y, int64_t n, ilw_stream_t stream);

/* Integer top-K (the two-stage query selection of Sec. 3.1.2): for each of `rows` rows of S (int32, leading dimension
 * lds), the K largest of its first N values in decreasing order, equal values ordered by
 * increasing index.  vals, idx int32 [rows, K] device.  1 <= K <= N <= 16384. */
int ilwdetr_topk(const int32_t *S, int64_t lds, int32_t rows, int32_t N, int32_t K, int32_t *vals,
                 int32_t *idx, ilw_stream_t stream);

/* Row gather (the selected tokens' memory rows and anchors of the two-stage selection, Sec. 3.1.2):
 * dst row i = src row idx[i], i < n (row_bytes bytes each; leading dimensions in
 * bytes).  src, dst, idx device; row_bytes, src_ld, dst_ld multiples of 4, pointers 4-byte
 * aligned.  An index outside [0, src_rows) gives a zero row and is reported by the next
 * ilwdetr_device_status. */
int ilwdetr_gather_rows(const void *src, int64_t src_ld, int64_t src_rows, const int32_t *idx, int64_t n,
                        int64_t row_bytes, void *dst, int64_t dst_ld, ilw_stream_t stream);

#ifdef __cplusplus
}
#endif
#endif
