// abi.cu -- the extern "C" entry points declared in include/ilwdetr.h: argument validation,
// integer parameter preparation (ShiftExp reciprocal constants) and kernel dispatch.
// Nothing here computes on the host: every step of the path runs in the kernels.
#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <string>

#include "ilw_kernels.h"
#include "ilwdetr.h"

namespace {

thread_local std::string g_err;

int fail(int code, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    g_err = buf;
    return code;
}

int cuda_status(cudaError_t e, const char *what) {
    if (e == cudaSuccess) return ILW_OK;
    return fail(ILW_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned(const void *p, size_t a) { return ((uintptr_t)p % a) == 0; }

int check_shiftmax(const ilw_shiftmax_t *p) {
    if (!p) return fail(ILW_ERR_INVALID_ARG, "shiftmax parameters are NULL");
    if (p->I0 < 1 || p->I0 >= (1 << 15))
        return fail(ILW_ERR_INVALID_ARG, "shiftmax I0=%d outside [1, 2^15)", p->I0);
    if (p->k_inter < 0 || p->k_inter > 16)
        return fail(ILW_ERR_INVALID_ARG, "shiftmax k_inter=%d outside [0, 16]", p->k_inter);
    if (((int64_t)p->I0 << p->k_inter) >= ((int64_t)1 << 31))
        return fail(ILW_ERR_INVALID_ARG, "shiftmax I0 * 2^k_inter must be < 2^31");
    if (p->k_out < 1 || p->k_out > 8) return fail(ILW_ERR_INVALID_ARG, "shiftmax k_out=%d outside [1, 8]", p->k_out);
    if (p->s_d > 31) return fail(ILW_ERR_INVALID_ARG, "static s_d=%d > 31", p->s_d);
    if (p->m_p < 0 || p->m_p > 31 || p->M_hw < 1 || p->M_hw > 31)
        return fail(ILW_ERR_INVALID_ARG, "m_p=%d / M_hw=%d out of range", p->m_p, p->M_hw);
    return ILW_OK;
}

int check_gelu(const ilw_gelu_t *p) {
    if (!p) return fail(ILW_ERR_INVALID_ARG, "gelu parameters are NULL");
    if (p->I0 < 1 || p->I0 >= (1 << 15)) return fail(ILW_ERR_INVALID_ARG, "gelu I0=%d outside [1, 2^15)", p->I0);
    if (p->k_inter < 0 || p->k_inter > 16)
        return fail(ILW_ERR_INVALID_ARG, "gelu k_inter=%d outside [0, 16]", p->k_inter);
    if (((int64_t)p->I0 << (p->k_inter + 1)) >= ((int64_t)1 << 31))
        return fail(ILW_ERR_INVALID_ARG, "gelu I0 * 2^(k_inter+1) must be < 2^31");
    if (p->k_out < 1 || p->k_out > 8) return fail(ILW_ERR_INVALID_ARG, "gelu k_out=%d outside [1, 8]", p->k_out);
    return ILW_OK;
}

ilw::ShiftmaxC make_smx(const ilw_shiftmax_t &p) {
    ilw::ShiftmaxC c;
    c.se = ilw::make_shiftexp(p.I0, p.k_inter);
    c.s_d = p.s_d < 0 ? -1 : p.s_d;
    c.m_p = p.m_p;
    c.M_hw = p.M_hw;
    c.k_out = p.k_out;
    return c;
}

int check_rq_scalar(int32_t s, const char *what) {
    if (s < 1 || s > 62) return fail(ILW_ERR_INVALID_ARG, "%s shift=%d outside [1, 62]", what, s);
    return ILW_OK;
}

int gemm_common(const int8_t *A, int64_t lda, const void *Wp, int32_t M, int32_t N, int32_t K) {
    if (M < 0 || N < 0 || K < 1) return fail(ILW_ERR_INVALID_ARG, "bad GEMM sizes M=%d N=%d K=%d", M, N, K);
    if (K % 16) return fail(ILW_ERR_UNSUPPORTED, "K=%d must be a multiple of 16", K);
    if (M == 0 || N == 0) return ILW_OK;
    if (!A || !Wp) return fail(ILW_ERR_INVALID_ARG, "GEMM operand is NULL");
    if (lda < K || lda % 16 || !aligned(A, 16)) return fail(ILW_ERR_INVALID_ARG, "A must be 16-byte aligned with lda >= K, lda %% 16 == 0");
    if (!aligned(Wp, 256)) return fail(ILW_ERR_INVALID_ARG, "packed weight must be 256-byte aligned");
    if (K > (1 << 20)) return fail(ILW_ERR_UNSUPPORTED, "K too large");
    return ILW_OK;
}

}  // namespace

int ilw::report_error(int code, const char *msg) { return fail(code, "%s", msg); }

extern "C" {

const char *ilwdetr_version(void) { return "ilwdetr 0.1 sm_103a"; }
const char *ilwdetr_last_error(void) { return g_err.c_str(); }

int ilwdetr_device_status(ilw_stream_t stream) {
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_status(e, "cudaStreamSynchronize");
    int v = 0;
    e = ilw::read_and_clear_status(&v);
    if (e != cudaSuccess) return cuda_status(e, "read device status");
    if (v) return fail(ILW_ERR_TIMEOUT, "a kernel's bounded wait expired (code %d)", v);
    return ILW_OK;
}

size_t ilwdetr_packed_weight_bytes(int32_t N, int32_t K) {
    if (N < 0 || K < 0) return 0;
    return ilw::packed_weight_bytes(N, K);
}

int ilwdetr_pack_weight(const int8_t *W, int32_t N, int32_t K, void *packed, ilw_stream_t stream) {
    if (N < 0 || K < 1 || K % 16) return fail(ILW_ERR_INVALID_ARG, "pack: bad sizes N=%d K=%d (K %% 16 == 0)", N, K);
    if (N == 0) return ILW_OK;
    if (!W || !packed) return fail(ILW_ERR_INVALID_ARG, "pack: NULL pointer");
    if (!aligned(packed, 256)) return fail(ILW_ERR_INVALID_ARG, "pack: output must be 256-byte aligned");
    return cuda_status(ilw::launch_pack_weight(W, N, K, packed, (cudaStream_t)stream), "pack_weight");
}

int ilwdetr_gemm_requant(const int8_t *A, int64_t lda, const void *Wp, const int32_t *bias,
                         const int32_t *mult, const int32_t *shift, int32_t M, int32_t N, int32_t K,
                         int32_t out_bits, void *C, int64_t ldc, const ilw_residual_t *res,
                         ilw_stream_t stream) {
    int rc = gemm_common(A, lda, Wp, M, N, K);
    if (rc) return rc;
    if (out_bits != 8 && out_bits != 16 && out_bits != 32 && out_bits != ILW_I8_IN_F16)
        return fail(ILW_ERR_INVALID_ARG, "out_bits=%d must be 8, 16, 32 or ILW_I8_IN_F16", out_bits);
    if (M == 0 || N == 0) return ILW_OK;
    if (!C || ldc < N) return fail(ILW_ERR_INVALID_ARG, "C is NULL or ldc < N");
    if (out_bits != 32 && (!mult || !shift)) return fail(ILW_ERR_INVALID_ARG, "mult/shift are NULL");
    if (res && out_bits != 32) {
        if (!res->x || res->rows < 1 || res->ldx < N) return fail(ILW_ERR_INVALID_ARG, "bad residual");
        if ((rc = check_rq_scalar(res->shift, "residual"))) return rc;
    }
    ilw::GemmProblem gp{};
    gp.M = M;
    gp.N = N;
    gp.nb = 1;
    gp.branch_rq = false;
    gp.br[0] = {A, lda, ilw::packed_i8(Wp), ilw::packed_f16(Wp, N, K), K, 0, 0};
    ilw::EpiParams ep{};
    ep.kind = ilw::EPI_REQUANT;
    ep.bias = bias;
    ep.mult = mult;
    ep.shift = shift;
    ep.out_bits = out_bits;
    ep.C = C;
    ep.ldc = ldc;
    if (res && out_bits != 32) {
        ep.res = res->x;
        ep.ldr = res->ldx;
        ep.res_rows = res->rows;
        ep.m_r = res->mult;
        ep.s_r = res->shift;
    }
    return cuda_status(ilw::launch_gemm(gp, ep, (cudaStream_t)stream), "gemm_requant");
}

int ilwdetr_gemm_gelu(const int8_t *A, int64_t lda, const void *Wp, const int32_t *bias,
                      const int32_t *mult, const int32_t *shift, int32_t M, int32_t N, int32_t K,
                      const ilw_gelu_t *gelu, int32_t m_g, int32_t s_g, int8_t *H, int64_t ldh,
                      ilw_stream_t stream) {
    int rc = gemm_common(A, lda, Wp, M, N, K);
    if (rc) return rc;
    if ((rc = check_gelu(gelu))) return rc;
    if ((rc = check_rq_scalar(s_g, "gelu output"))) return rc;
    if (M == 0 || N == 0) return ILW_OK;
    if (!H || ldh < N || !mult || !shift) return fail(ILW_ERR_INVALID_ARG, "gemm_gelu: bad output or NULL mult/shift");
    ilw::GemmProblem gp{};
    gp.M = M;
    gp.N = N;
    gp.nb = 1;
    gp.br[0] = {A, lda, ilw::packed_i8(Wp), ilw::packed_f16(Wp, N, K), K, 0, 0};
    ilw::EpiParams ep{};
    ep.kind = ilw::EPI_GELU;
    ep.bias = bias;
    ep.mult = mult;
    ep.shift = shift;
    ep.C = H;
    ep.ldc = ldh;
    ep.gelu = ilw::make_gelu(*gelu);
    ep.m_g = m_g;
    ep.s_g = s_g;
    return cuda_status(ilw::launch_gemm(gp, ep, (cudaStream_t)stream), "gemm_gelu");
}

int ilwdetr_split_conv(const int8_t *const *X, const int64_t *ldx, int32_t nb, int32_t M,
                       const int32_t *Kb, const void *const *Wp, const int32_t *m_b,
                       const int32_t *s_b, const int32_t *bias, const int32_t *mult,
                       const int32_t *shift, int32_t N, int8_t *Y, int64_t ldy,
                       ilw_stream_t stream) {
    if (nb < 1 || nb > ilw::kMaxBranches) return fail(ILW_ERR_INVALID_ARG, "nb=%d outside [1, 8]", nb);
    if (!X || !ldx || !Kb || !Wp || !m_b || !s_b) return fail(ILW_ERR_INVALID_ARG, "split_conv: NULL host array");
    if (M < 0 || N < 0) return fail(ILW_ERR_INVALID_ARG, "split_conv: bad sizes");
    ilw::GemmProblem gp{};
    gp.M = M;
    gp.N = N;
    gp.nb = nb;
    gp.branch_rq = true;
    for (int b = 0; b < nb; ++b) {
        int rc = gemm_common(X[b], ldx[b], Wp[b], M, N, Kb[b]);
        if (rc) return rc;
        if ((rc = check_rq_scalar(s_b[b], "branch"))) return rc;
        if (Kb[b] > 1024) return fail(ILW_ERR_UNSUPPORTED, "split_conv: branch %d has K=%d > 1024", b, Kb[b]);
        if (m_b[b] < 0 || (s_b[b] <= 31 && (int64_t)m_b[b] > ((int64_t)1 << s_b[b])))
            return fail(ILW_ERR_INVALID_ARG, "branch %d: ratio m_b / 2^s_b must be in [0, 1]", b);
        gp.br[b] = {X[b], ldx[b], ilw::packed_i8(Wp[b]), ilw::packed_f16(Wp[b], N, Kb[b]), Kb[b], m_b[b], s_b[b]};
    }
    if (M == 0 || N == 0) return ILW_OK;
    if (!Y || ldy < N || !mult || !shift) return fail(ILW_ERR_INVALID_ARG, "split_conv: bad output or NULL mult/shift");
    ilw::EpiParams ep{};
    ep.kind = ilw::EPI_REQUANT;
    ep.bias = bias;
    ep.mult = mult;
    ep.shift = shift;
    ep.out_bits = 8;
    ep.C = Y;
    ep.ldc = ldy;
    return cuda_status(ilw::launch_gemm(gp, ep, (cudaStream_t)stream), "split_conv");
}

int ilwdetr_shiftmax_rows(const int32_t *X, int64_t ldx, int64_t rows, int32_t len,
                          const ilw_shiftmax_t *p, uint8_t *P, int64_t ldp, ilw_stream_t stream) {
    int rc = check_shiftmax(p);
    if (rc) return rc;
    if (rows < 0 || len < 0) return fail(ILW_ERR_INVALID_ARG, "shiftmax_rows: negative size");
    if (rows == 0 || len == 0) return ILW_OK;
    if (!X || !P || ldx < len || ldp < len) return fail(ILW_ERR_INVALID_ARG, "shiftmax_rows: NULL pointer or ld < len");
    if (!aligned(X, 4)) return fail(ILW_ERR_INVALID_ARG, "shiftmax_rows: X must be 4-byte aligned");
    return cuda_status(ilw::launch_shiftmax_rows(X, ldx, rows, len, make_smx(*p), P, ldp, (cudaStream_t)stream),
                       "shiftmax_rows");
}

int ilwdetr_sdshiftgelu(const int32_t *X, int32_t *Y, int64_t n, const ilw_gelu_t *p, ilw_stream_t stream) {
    int rc = check_gelu(p);
    if (rc) return rc;
    if (n < 0) return fail(ILW_ERR_INVALID_ARG, "sdshiftgelu: n < 0");
    if (n == 0) return ILW_OK;
    if (!X || !Y || !aligned(X, 4) || !aligned(Y, 4)) return fail(ILW_ERR_INVALID_ARG, "sdshiftgelu: NULL or misaligned");
    return cuda_status(ilw::launch_sdshiftgelu(X, Y, n, ilw::make_gelu(*p), (cudaStream_t)stream), "sdshiftgelu");
}

int ilwdetr_int_layernorm(const void *X, int32_t in_bits, int64_t ldx, int64_t rows, int32_t C,
                          const int32_t *beta, const int32_t *mult, const int32_t *shift,
                          int32_t iters, void *Y, int32_t out_bits, int64_t ldy, ilw_stream_t stream) {
    if (in_bits != 16 && in_bits != 32) return fail(ILW_ERR_INVALID_ARG, "in_bits=%d must be 16 or 32", in_bits);
    if (out_bits != 8 && out_bits != 16) return fail(ILW_ERR_INVALID_ARG, "out_bits=%d must be 8 or 16", out_bits);
    if (C < 1 || C > 4096) return fail(ILW_ERR_UNSUPPORTED, "C=%d outside [1, 4096]", C);
    if (rows < 0 || iters < 0 || iters > 64) return fail(ILW_ERR_INVALID_ARG, "bad rows / iters");
    if (rows == 0) return ILW_OK;
    if (!X || !Y || !beta || !mult || !shift || ldx < C || ldy < C)
        return fail(ILW_ERR_INVALID_ARG, "int_layernorm: NULL pointer or ld < C");
    ilw::LnParams lp{X, in_bits, ldx, rows, C, beta, mult, shift, iters, Y, out_bits, ldy};
    return cuda_status(ilw::launch_layernorm(lp, (cudaStream_t)stream), "int_layernorm");
}

static int attn_params(ilw::AttnParams &ap, const void *Q, const void *K, const void *V, int64_t ld_qkv,
                       int32_t qkv_form, int32_t B, int32_t T, int32_t H, int32_t dh, int32_t win_side,
                       const ilw_shiftmax_t *p, int32_t m_o, int32_t s_o, int8_t *O, int64_t ld_o) {
    int rc = check_shiftmax(p);
    if (rc) return rc;
    if ((rc = check_rq_scalar(s_o, "attention output"))) return rc;
    if (B < 0 || T < 0 || H < 1) return fail(ILW_ERR_INVALID_ARG, "attention: bad sizes");
    if (dh != 32 && dh != 64) return fail(ILW_ERR_UNSUPPORTED, "attention: dh=%d must be 32 or 64", dh);
    if (!Q || !K || !V || !O) return fail(ILW_ERR_INVALID_ARG, "attention: NULL pointer");
    if (qkv_form != 8 && qkv_form != ILW_I8_IN_F16)
        return fail(ILW_ERR_INVALID_ARG, "attention: qkv_form=%d must be 8 or ILW_I8_IN_F16", qkv_form);
    const int64_t esz = qkv_form == 8 ? 1 : 2;
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || (ld_qkv * esz) % 16 || ld_qkv < (int64_t)H * dh)
        return fail(ILW_ERR_INVALID_ARG, "attention: q/k/v must be 16-byte aligned with 16-byte aligned rows");
    if (ld_o < (int64_t)H * dh) return fail(ILW_ERR_INVALID_ARG, "attention: ld_o < H*dh");
    ap = {};
    ap.Q = Q; ap.K = K; ap.V = V; ap.ld_qkv = ld_qkv;
    ap.qkv_f16 = qkv_form == ILW_I8_IN_F16 ? 1 : 0;
    ap.B = B; ap.T = T; ap.H = H; ap.dh = dh;
    ap.nw = win_side <= 1 ? 1 : win_side;
    ap.grid_side = 0;
    if (ap.nw > 1) {
        int g = 0;
        while ((int64_t)(g + 1) * (g + 1) <= T) ++g;
        if ((int64_t)g * g != T || g % ap.nw)
            return fail(ILW_ERR_INVALID_ARG, "window attention: T=%d is not a square grid divisible by %d", T, ap.nw);
        ap.grid_side = g;
    }
    ap.smx = make_smx(*p);
    ap.m_o = m_o; ap.s_o = s_o;
    ap.O = O; ap.ld_o = ld_o;
    return ILW_OK;
}

int ilwdetr_shiftmax_attn(const void *Q, const void *K, const void *V, int64_t ld_qkv, int32_t qkv_form,
                          int32_t B, int32_t T, int32_t H, int32_t dh, int32_t win_side, const ilw_shiftmax_t *p,
                          int32_t m_o, int32_t s_o, int8_t *O, int64_t ld_o, ilw_stream_t stream) {
    if (B == 0 || T == 0) return ILW_OK;
    ilw::AttnParams ap;
    int rc = attn_params(ap, Q, K, V, ld_qkv, qkv_form, B, T, H, dh, win_side, p, m_o, s_o, O, ld_o);
    if (rc) return rc;
    return cuda_status(ilw::launch_attention(ap, (cudaStream_t)stream), "shiftmax_attn");
}

int ilwdetr_deform_attn(const int8_t *value, const int32_t *level_hw, int32_t L, const int32_t *ref_q16,
                        const int32_t *off_q8, const uint8_t *w, int32_t B, int32_t Q, int32_t H, int32_t P,
                        int32_t dh, int32_t m, int32_t s, int8_t *out, ilw_stream_t stream) {
    if (L < 1 || L > 8 || !level_hw) return fail(ILW_ERR_INVALID_ARG, "deform: L=%d outside [1, 8]", L);
    if (B < 0 || Q < 0 || H < 1 || P < 1 || dh < 4 || dh % 4) return fail(ILW_ERR_INVALID_ARG, "deform: bad sizes (dh %% 4 == 0)");
    int rc = check_rq_scalar(s, "deform output");
    if (rc) return rc;
    if (B == 0 || Q == 0) return ILW_OK;
    if (!value || !ref_q16 || !off_q8 || !w || !out) return fail(ILW_ERR_INVALID_ARG, "deform: NULL pointer");
    if (!aligned(value, 4) || !aligned(out, 4)) return fail(ILW_ERR_INVALID_ARG, "deform: value/out must be 4-byte aligned");
    ilw::DeformParams dp{};
    dp.value = value;
    dp.L = L;
    int64_t st = 0;
    for (int l = 0; l < L; ++l) {
        if (level_hw[2 * l] < 1 || level_hw[2 * l + 1] < 1) return fail(ILW_ERR_INVALID_ARG, "deform: level %d has no pixels", l);
        dp.lh[l] = level_hw[2 * l];
        dp.lw[l] = level_hw[2 * l + 1];
        dp.lstart[l] = st;
        st += (int64_t)dp.lh[l] * dp.lw[l];
    }
    dp.S_total = st;
    dp.ref = ref_q16; dp.off = off_q8; dp.w = w;
    dp.B = B; dp.Q = Q; dp.H = H; dp.P = P; dp.dh = dh;
    dp.m = m; dp.s = s;
    dp.out = out;
    return cuda_status(ilw::launch_deform(dp, (cudaStream_t)stream), "deform_attn");
}

// ------------------------------------------------------------------ patch embedding
static size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

size_t ilwdetr_patch_embed_workspace_bytes(int32_t B, int32_t Cin, int32_t Hh, int32_t Ww, int32_t p) {
    if (B < 0 || Cin < 1 || p < 1 || Hh < 0 || Ww < 0) return 0;
    return align256((size_t)B * (Hh / p) * (Ww / p) * Cin * p * p);
}

int ilwdetr_patch_embed(const int8_t *img, int32_t B, int32_t Cin, int32_t Hh, int32_t Ww, int32_t p,
                        const void *Wp, const int32_t *bias, const int32_t *mult, const int32_t *shift,
                        int32_t d, const int16_t *pos, int32_t m_pos, int32_t s_pos, int16_t *x0,
                        void *workspace, size_t workspace_bytes, ilw_stream_t stream) {
    if (B < 0 || Cin < 1 || p < 16 || p % 16 || Hh < p || Ww < p || Hh % p || Ww % p || Ww % 16 || d < 1)
        return fail(ILW_ERR_UNSUPPORTED, "patch_embed: needs p %% 16 == 0, p | H, p | W (p=%d H=%d W=%d)", p, Hh, Ww);
    if (B == 0) return ILW_OK;
    if (!img || !aligned(img, 16) || !x0) return fail(ILW_ERR_INVALID_ARG, "patch_embed: NULL or misaligned image");
    if (!workspace || !aligned(workspace, 256) ||
        workspace_bytes < ilwdetr_patch_embed_workspace_bytes(B, Cin, Hh, Ww, p))
        return fail(ILW_ERR_INVALID_ARG, "patch_embed: workspace too small or misaligned");
    const int32_t T = (Hh / p) * (Ww / p), K = Cin * p * p;
    int8_t *A = (int8_t *)workspace;
    cudaError_t e = ilw::launch_patchify(img, B, Cin, Hh, Ww, p, A, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_status(e, "patchify");
    if (pos) {
        ilw_residual_t r{pos, d, T, m_pos, s_pos};
        return ilwdetr_gemm_requant(A, K, Wp, bias, mult, shift, B * T, d, K, 16, x0, d, &r, stream);
    }
    return ilwdetr_gemm_requant(A, K, Wp, bias, mult, shift, B * T, d, K, 16, x0, d, nullptr, stream);
}

// ------------------------------------------------------------------ encoder block

size_t ilwdetr_block_workspace_bytes(int32_t B, int32_t T, int32_t d, int32_t F) {
    if (B < 0 || T < 0 || d < 0 || F < 0) return 0;
    size_t M = (size_t)B * T;
    return align256(M * d) /*a1*/ + align256(M * 3 * d * 2) /*qkv (fp16)*/ + align256(M * d) /*O*/ +
           align256(M * d * 2) /*x1*/ + align256(M * d) /*a2*/ + align256(M * F) /*h*/;
}

int ilwdetr_block_forward(const ilw_block_params_t *p, const int16_t *x, int16_t *y, int32_t B, int32_t T,
                          void *workspace, size_t workspace_bytes, ilw_stream_t stream) {
    if (!p || p->struct_size != sizeof(ilw_block_params_t))
        return fail(ILW_ERR_INVALID_ARG, "block params NULL or struct_size mismatch");
    const int32_t d = p->d, H = p->H, F = p->F;
    if (d < 16 || d % 16 || H < 1 || d % H || F < 16 || F % 16)
        return fail(ILW_ERR_INVALID_ARG, "block: d=%d H=%d F=%d (d, F multiples of 16, H | d)", d, H, F);
    if (B < 0 || T < 0) return fail(ILW_ERR_INVALID_ARG, "block: negative sizes");
    if (B == 0 || T == 0) return ILW_OK;
    if (!x || !y || x == y) return fail(ILW_ERR_INVALID_ARG, "block: x/y NULL or aliased");
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < ilwdetr_block_workspace_bytes(B, T, d, F))
        return fail(ILW_ERR_INVALID_ARG, "block: workspace NULL, misaligned or smaller than %zu bytes",
                    ilwdetr_block_workspace_bytes(B, T, d, F));
    const int32_t M = B * T;
    char *ws = (char *)workspace;
    int8_t *a1 = (int8_t *)ws; ws += align256((size_t)M * d);
    __half *qkv = (__half *)ws; ws += align256((size_t)M * 3 * d * 2);  // q|k|v as fp16 (ILW_I8_IN_F16)
    int8_t *o = (int8_t *)ws; ws += align256((size_t)M * d);
    int16_t *x1 = (int16_t *)ws; ws += align256((size_t)M * d * 2);
    int8_t *a2 = (int8_t *)ws; ws += align256((size_t)M * d);
    int8_t *hbuf = (int8_t *)ws;
    int rc;
    if ((rc = ilwdetr_int_layernorm(x, 16, d, M, d, p->ln1_beta, p->ln1_mult, p->ln1_shift, p->ln_iters, a1, 8, d, stream)))
        return rc;
    if ((rc = ilwdetr_gemm_requant(a1, d, p->w_qkv, p->b_qkv, p->m_qkv, p->s_qkv, M, 3 * d, d, ILW_I8_IN_F16, qkv, 3 * d,
                                   nullptr, stream)))
        return rc;
    if ((rc = ilwdetr_shiftmax_attn(qkv, qkv + d, qkv + 2 * d, 3 * d, ILW_I8_IN_F16, B, T, H, d / H, p->win_side, &p->smx, p->m_o,
                                    p->s_o, o, d, stream)))
        return rc;
    ilw_residual_t r1{x, d, M, p->m_r1, p->s_r1};
    if ((rc = ilwdetr_gemm_requant(o, d, p->w_proj, p->b_proj, p->m_proj, p->s_proj, M, d, d, 16, x1, d, &r1, stream)))
        return rc;
    if ((rc = ilwdetr_int_layernorm(x1, 16, d, M, d, p->ln2_beta, p->ln2_mult, p->ln2_shift, p->ln_iters, a2, 8, d, stream)))
        return rc;
    if ((rc = ilwdetr_gemm_gelu(a2, d, p->w_fc1, p->b_fc1, p->m_fc1, p->s_fc1, M, F, d, &p->gelu, p->m_g, p->s_g, hbuf, F,
                                stream)))
        return rc;
    ilw_residual_t r2{x1, d, M, p->m_r2, p->s_r2};
    return ilwdetr_gemm_requant(hbuf, F, p->w_fc2, p->b_fc2, p->m_fc2, p->s_fc2, M, d, F, 16, y, d, &r2, stream);
}

}  // extern "C"
