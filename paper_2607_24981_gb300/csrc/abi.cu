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

// Composite entry points (the patch embedding, the encoder block, the decoder layer) run their
// steps twice: first with every launch suppressed, which checks each step's arguments with the
// step's own validation, then for real; so an argument error in a later step is reported before
// the first launch.  Each entry point's launch is skipped (ILW_OK) while g_check_only is set;
// ilwdetr_validate_only sets it for the calling thread until it is cleared again.
thread_local bool g_check_only = false;
struct CheckPass {
    CheckPass() { g_check_only = true; }
    ~CheckPass() { g_check_only = false; }
};
template <typename Body> int checked_then_run(Body body) {
    if (g_check_only) return body();  // inside another composite's checking pass
    {
        CheckPass pass;
        if (const int rc = body()) return rc;
    }
    return body();
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
bool ilw::validate_only() { return g_check_only; }

extern "C" {

const char *ilwdetr_version(void) { return "ilwdetr 0.1 sm_103a"; }
const char *ilwdetr_last_error(void) { return g_err.c_str(); }

int ilwdetr_device_status(ilw_stream_t stream) {
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_status(e, "cudaStreamSynchronize");
    int v = 0;
    e = ilw::read_and_clear_status(&v);
    if (e != cudaSuccess) return cuda_status(e, "read device status");
    if (v == ilw::kStatusBadIndex) return fail(ILW_ERR_INVALID_ARG, "a gather index lay outside its source rows");
    if (v) return fail(ILW_ERR_TIMEOUT, "a kernel's bounded wait expired (code %d)", v);
    return ILW_OK;
}

int ilwdetr_validate_only(int32_t on) {
    g_check_only = on != 0;
    return ILW_OK;
}

int ilwdetr_debug_gemm_wait(int32_t skip_load, int64_t wait_cycles) {
    if (skip_load < -1 || wait_cycles < 0) return fail(ILW_ERR_INVALID_ARG, "debug_gemm_wait: skip_load >= -1, wait_cycles >= 0");
    ilw::gemm_set_debug_wait(skip_load, (long long)wait_cycles);
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
    if (g_check_only) return ILW_OK;
    return cuda_status(ilw::launch_pack_weight(W, N, K, packed, (cudaStream_t)stream), "pack_weight");
}

namespace {
// The common path of the GEMM entry points.
int gemm_impl(const void *A, int32_t a_form, int64_t lda, const void *Wp, const int32_t *bias, const int32_t *mult,
              const int32_t *shift, int32_t M, int32_t N, int32_t K, int32_t epilogue, int32_t out_bits, void *C,
              int64_t ldc, const ilw_residual_t *res, const ilw_gelu_t *gelu, int32_t m_g, int32_t s_g,
              ilw_stream_t stream, const char *what) {
    if (a_form != 8 && a_form != ILW_I8_IN_F16)
        return fail(ILW_ERR_INVALID_ARG, "%s: a_form=%d must be 8 or ILW_I8_IN_F16", what, a_form);
    int rc;
    if (a_form == 8) {
        if ((rc = gemm_common((const int8_t *)A, lda, Wp, M, N, K))) return rc;
    } else {
        if (M < 0 || N < 0 || K < 1) return fail(ILW_ERR_INVALID_ARG, "bad GEMM sizes M=%d N=%d K=%d", M, N, K);
        if (K % 16) return fail(ILW_ERR_UNSUPPORTED, "K=%d must be a multiple of 16", K);
        if (M == 0 || N == 0) return ILW_OK;
        if (!A || !Wp) return fail(ILW_ERR_INVALID_ARG, "GEMM operand is NULL");
        if (lda < K || lda % 8 || !aligned(A, 16))
            return fail(ILW_ERR_INVALID_ARG, "fp16 A must be 16-byte aligned with lda >= K, lda %% 8 == 0");
        if (!aligned(Wp, 256)) return fail(ILW_ERR_INVALID_ARG, "packed weight must be 256-byte aligned");
        if (K > (1 << 20)) return fail(ILW_ERR_UNSUPPORTED, "K too large");
    }
    if (epilogue == ILW_EPI_GELU) {
        if ((rc = check_gelu(gelu))) return rc;
        if ((rc = check_rq_scalar(s_g, "gelu output"))) return rc;
        if (out_bits != 8 && out_bits != ILW_I8_IN_F16)
            return fail(ILW_ERR_INVALID_ARG, "%s: GELU out_bits=%d must be 8 or ILW_I8_IN_F16", what, out_bits);
    } else if (epilogue != ILW_EPI_REQUANT) {
        return fail(ILW_ERR_INVALID_ARG, "%s: epilogue=%d unknown", what, epilogue);
    } else if (out_bits != 8 && out_bits != 16 && out_bits != 32 && out_bits != ILW_I8_IN_F16) {
        return fail(ILW_ERR_INVALID_ARG, "out_bits=%d must be 8, 16, 32 or ILW_I8_IN_F16", out_bits);
    }
    if (M == 0 || N == 0) return ILW_OK;
    if (!C || ldc < N) return fail(ILW_ERR_INVALID_ARG, "C is NULL or ldc < N");
    if (out_bits != 32 && (!mult || !shift)) return fail(ILW_ERR_INVALID_ARG, "mult/shift are NULL");
    const bool use_res = res && epilogue == ILW_EPI_REQUANT && out_bits != 32;
    if (use_res) {
        if (!res->x || res->rows < 1 || res->ldx < N) return fail(ILW_ERR_INVALID_ARG, "bad residual");
        if ((rc = check_rq_scalar(res->shift, "residual"))) return rc;
    }
    ilw::GemmProblem gp{};
    gp.M = M;
    gp.N = N;
    gp.nb = 1;
    gp.branch_rq = false;
    gp.a_f16 = a_form == ILW_I8_IN_F16;
    gp.br[0] = {(const int8_t *)A, lda, ilw::packed_i8(Wp), ilw::packed_f16(Wp, N, K), K, 0, 0};
    ilw::EpiParams ep{};
    ep.kind = epilogue == ILW_EPI_GELU ? ilw::EPI_GELU : ilw::EPI_REQUANT;
    ep.bias = bias;
    ep.mult = mult;
    ep.shift = shift;
    ep.out_bits = out_bits;
    ep.C = C;
    ep.ldc = ldc;
    if (use_res) {
        ep.res = res->x;
        ep.ldr = res->ldx;
        ep.res_rows = res->rows;
        ep.m_r = res->mult;
        ep.s_r = res->shift;
    }
    if (epilogue == ILW_EPI_GELU) {
        ep.gelu = ilw::make_gelu(*gelu);
        ep.m_g = m_g;
        ep.s_g = s_g;
    }
    if (g_check_only) return ILW_OK;
    return cuda_status(ilw::launch_gemm(gp, ep, (cudaStream_t)stream), what);
}
}  // namespace

int ilwdetr_gemm_requant(const int8_t *A, int64_t lda, const void *Wp, const int32_t *bias,
                         const int32_t *mult, const int32_t *shift, int32_t M, int32_t N, int32_t K,
                         int32_t out_bits, void *C, int64_t ldc, const ilw_residual_t *res,
                         ilw_stream_t stream) {
    return gemm_impl(A, 8, lda, Wp, bias, mult, shift, M, N, K, ILW_EPI_REQUANT, out_bits, C, ldc, res, nullptr, 0,
                     0, stream, "gemm_requant");
}

int ilwdetr_gemm_gelu(const int8_t *A, int64_t lda, const void *Wp, const int32_t *bias,
                      const int32_t *mult, const int32_t *shift, int32_t M, int32_t N, int32_t K,
                      const ilw_gelu_t *gelu, int32_t m_g, int32_t s_g, int8_t *H, int64_t ldh,
                      ilw_stream_t stream) {
    return gemm_impl(A, 8, lda, Wp, bias, mult, shift, M, N, K, ILW_EPI_GELU, 8, H, ldh, nullptr, gelu, m_g, s_g,
                     stream, "gemm_gelu");
}

int ilwdetr_gemm(const ilw_gemm_t *g, ilw_stream_t stream) {
    if (!g || g->struct_size != sizeof(ilw_gemm_t)) return fail(ILW_ERR_INVALID_ARG, "gemm: NULL or struct_size mismatch");
    return gemm_impl(g->A, g->a_form, g->lda, g->Wp, g->bias, g->mult, g->shift, g->M, g->N, g->K, g->epilogue,
                     g->out_bits, g->C, g->ldc, g->res, g->gelu, g->m_g, g->s_g, stream, "gemm");
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
    if (g_check_only) return ILW_OK;
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
    if (g_check_only) return ILW_OK;
    return cuda_status(ilw::launch_shiftmax_rows(X, ldx, rows, len, make_smx(*p), P, ldp, (cudaStream_t)stream),
                       "shiftmax_rows");
}

int ilwdetr_sdshiftgelu(const int32_t *X, int32_t *Y, int64_t n, const ilw_gelu_t *p, ilw_stream_t stream) {
    int rc = check_gelu(p);
    if (rc) return rc;
    if (n < 0) return fail(ILW_ERR_INVALID_ARG, "sdshiftgelu: n < 0");
    if (n == 0) return ILW_OK;
    if (!X || !Y || !aligned(X, 4) || !aligned(Y, 4)) return fail(ILW_ERR_INVALID_ARG, "sdshiftgelu: NULL or misaligned");
    if (g_check_only) return ILW_OK;
    return cuda_status(ilw::launch_sdshiftgelu(X, Y, n, ilw::make_gelu(*p), (cudaStream_t)stream), "sdshiftgelu");
}

int ilwdetr_int_layernorm(const void *X, int32_t in_bits, int64_t ldx, int64_t rows, int32_t C,
                          const int32_t *beta, const int32_t *mult, const int32_t *shift,
                          int32_t iters, void *Y, int32_t out_bits, int64_t ldy, ilw_stream_t stream) {
    if (in_bits != 16 && in_bits != 32) return fail(ILW_ERR_INVALID_ARG, "in_bits=%d must be 16 or 32", in_bits);
    if (out_bits != 8 && out_bits != 16 && out_bits != ILW_I8_IN_F16)
        return fail(ILW_ERR_INVALID_ARG, "out_bits=%d must be 8, 16 or ILW_I8_IN_F16", out_bits);
    if (C < 1 || C > 4096) return fail(ILW_ERR_UNSUPPORTED, "C=%d outside [1, 4096]", C);
    if (rows < 0 || iters < 0 || iters > 64) return fail(ILW_ERR_INVALID_ARG, "bad rows / iters");
    if (rows == 0) return ILW_OK;
    if (!X || !Y || !beta || !mult || !shift || ldx < C || ldy < C)
        return fail(ILW_ERR_INVALID_ARG, "int_layernorm: NULL pointer or ld < C");
    ilw::LnParams lp{X, in_bits, ldx, rows, C, beta, mult, shift, iters, Y, out_bits, ldy};
    if (g_check_only) return ILW_OK;
    return cuda_status(ilw::launch_layernorm(lp, (cudaStream_t)stream), "int_layernorm");
}

static int attn_params(ilw::AttnParams &ap, const void *Q, const void *K, const void *V, int64_t ld_qkv,
                       int32_t qkv_form, int32_t B, int32_t T, int32_t H, int32_t dh, int32_t win_side,
                       const ilw_shiftmax_t *p, int32_t m_o, int32_t s_o, void *O, int32_t o_form,
                       int64_t ld_o) {
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
    if (o_form != 8 && o_form != ILW_I8_IN_F16)
        return fail(ILW_ERR_INVALID_ARG, "attention: o_form=%d must be 8 or ILW_I8_IN_F16", o_form);
    if (o_form == ILW_I8_IN_F16 && !aligned(O, 4)) return fail(ILW_ERR_INVALID_ARG, "attention: fp16 O misaligned");
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
    ap.O = O; ap.o_f16 = o_form == ILW_I8_IN_F16 ? 1 : 0; ap.ld_o = ld_o;
    return ILW_OK;
}

int ilwdetr_shiftmax_attn(const void *Q, const void *K, const void *V, int64_t ld_qkv, int32_t qkv_form,
                          int32_t B, int32_t T, int32_t H, int32_t dh, int32_t win_side, const ilw_shiftmax_t *p,
                          int32_t m_o, int32_t s_o, void *O, int32_t o_form, int64_t ld_o, ilw_stream_t stream) {
    if (B == 0 || T == 0) return ILW_OK;
    ilw::AttnParams ap;
    int rc = attn_params(ap, Q, K, V, ld_qkv, qkv_form, B, T, H, dh, win_side, p, m_o, s_o, O, o_form, ld_o);
    if (rc) return rc;
    if (g_check_only) return ILW_OK;
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
    if (g_check_only) return ILW_OK;
    return cuda_status(ilw::launch_deform(dp, (cudaStream_t)stream), "deform_attn");
}

// ------------------------------------------------------------------ patch embedding
static size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

size_t ilwdetr_patch_embed_workspace_bytes(int32_t B, int32_t Cin, int32_t Hh, int32_t Ww, int32_t p) {
    if (B < 0 || Cin < 1 || p < 1 || Hh < 0 || Ww < 0) return 0;
    return align256((size_t)B * (Hh / p) * (Ww / p) * Cin * p * p * 2);  // patch matrix, fp16-carried int8
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
    __half *A = (__half *)workspace;  // the patch matrix as fp16-carried int8: the GEMM reads it directly
    return checked_then_run([&]() -> int {
        if (!g_check_only) {
            cudaError_t e = ilw::launch_patchify_f16(img, B, Cin, Hh, Ww, p, A, (cudaStream_t)stream);
            if (e != cudaSuccess) return cuda_status(e, "patchify");
        }
        ilw_residual_t r{pos, d, T, m_pos, s_pos};
        return gemm_impl(A, ILW_I8_IN_F16, K, Wp, bias, mult, shift, B * T, d, K, ILW_EPI_REQUANT, 16, x0, d,
                         pos ? &r : nullptr, nullptr, 0, 0, stream, "patch_embed");
    });
}

// ------------------------------------------------------------------ encoder block

size_t ilwdetr_block_workspace_bytes(int32_t B, int32_t T, int32_t d, int32_t F) {
    if (B < 0 || T < 0 || d < 0 || F < 0) return 0;
    size_t M = (size_t)B * T;
    // every int8 activation between kernels is carried in fp16 (the tensor cores' operand form)
    return align256(M * d * 2) /*a1*/ + align256(M * 3 * d * 2) /*qkv*/ + align256(M * d * 2) /*O*/ +
           align256(M * d * 2) /*x1 (int16)*/ + align256(M * d * 2) /*a2*/ + align256(M * F * 2) /*h*/;
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
    const int32_t F16 = ILW_I8_IN_F16;
    char *ws = (char *)workspace;
    __half *a1 = (__half *)ws; ws += align256((size_t)M * d * 2);
    __half *qkv = (__half *)ws; ws += align256((size_t)M * 3 * d * 2);
    __half *o = (__half *)ws; ws += align256((size_t)M * d * 2);
    int16_t *x1 = (int16_t *)ws; ws += align256((size_t)M * d * 2);
    __half *a2 = (__half *)ws; ws += align256((size_t)M * d * 2);
    __half *hbuf = (__half *)ws;
    return checked_then_run([&]() -> int {
        int rc;
        if ((rc = ilwdetr_int_layernorm(x, 16, d, M, d, p->ln1_beta, p->ln1_mult, p->ln1_shift, p->ln_iters, a1, F16, d, stream)))
            return rc;
        if ((rc = gemm_impl(a1, F16, d, p->w_qkv, p->b_qkv, p->m_qkv, p->s_qkv, M, 3 * d, d, ILW_EPI_REQUANT, F16, qkv, 3 * d,
                            nullptr, nullptr, 0, 0, stream, "block qkv")))
            return rc;
        if ((rc = ilwdetr_shiftmax_attn(qkv, qkv + d, qkv + 2 * d, 3 * d, F16, B, T, H, d / H, p->win_side, &p->smx, p->m_o,
                                        p->s_o, o, F16, d, stream)))
            return rc;
        ilw_residual_t r1{x, d, M, p->m_r1, p->s_r1};
        if ((rc = gemm_impl(o, F16, d, p->w_proj, p->b_proj, p->m_proj, p->s_proj, M, d, d, ILW_EPI_REQUANT, 16, x1, d, &r1,
                            nullptr, 0, 0, stream, "block proj")))
            return rc;
        if ((rc = ilwdetr_int_layernorm(x1, 16, d, M, d, p->ln2_beta, p->ln2_mult, p->ln2_shift, p->ln_iters, a2, F16, d, stream)))
            return rc;
        if ((rc = gemm_impl(a2, F16, d, p->w_fc1, p->b_fc1, p->m_fc1, p->s_fc1, M, F, d, ILW_EPI_GELU, F16, hbuf, F, nullptr,
                            &p->gelu, p->m_g, p->s_g, stream, "block fc1")))
            return rc;
        ilw_residual_t r2{x1, d, M, p->m_r2, p->s_r2};
        return gemm_impl(hbuf, F16, F, p->w_fc2, p->b_fc2, p->m_fc2, p->s_fc2, M, d, F, ILW_EPI_REQUANT, 16, y, d, &r2,
                         nullptr, 0, 0, stream, "block fc2");
    });
}

// ------------------------------------------------------------------ detector: projector, decoder

int ilwdetr_requant(const void *X, int32_t in_bits, int64_t ldx, int64_t rows, int32_t C, int32_t m1,
                    int32_t s1, const int16_t *Z, int64_t ldz, int64_t z_rows, int32_t m2, int32_t s2,
                    int32_t out_bits, void *Y, int64_t ldy, ilw_stream_t stream) {
    if (in_bits != 16 && in_bits != 32) return fail(ILW_ERR_INVALID_ARG, "requant: in_bits=%d must be 16 or 32", in_bits);
    if (out_bits != 8 && out_bits != 16 && out_bits != 32)
        return fail(ILW_ERR_INVALID_ARG, "requant: out_bits=%d must be 8, 16 or 32", out_bits);
    if (rows < 0 || C < 0 || C % 4) return fail(ILW_ERR_UNSUPPORTED, "requant: C=%d must be a multiple of 4", C);
    int rc;
    if ((rc = check_rq_scalar(s1, "requant"))) return rc;
    if (Z && (rc = check_rq_scalar(s2, "requant second term"))) return rc;
    if (rows == 0 || C == 0) return ILW_OK;
    const int64_t ib = in_bits / 8, ob = out_bits / 8;
    if (!X || !Y || ldx < C || ldy < C || !aligned(X, 4 * ib) || !aligned(Y, 4 * ob) || ldx % 4 || ldy % 4)
        return fail(ILW_ERR_INVALID_ARG, "requant: NULL, misaligned or short rows");
    if (Z && (z_rows < 1 || ldz < C || !aligned(Z, 8) || ldz % 4))
        return fail(ILW_ERR_INVALID_ARG, "requant: bad second term");
    ilw::RequantParams p{X, in_bits, ldx, rows, C, m1, s1, Z, ldz, Z ? z_rows : 1, m2, Z ? s2 : 1, out_bits, Y, ldy};
    if (g_check_only) return ILW_OK;
    return cuda_status(ilw::launch_requant(p, (cudaStream_t)stream), "requant");
}

int ilwdetr_resample_nearest(const int8_t *X, int64_t x_bstride, int32_t B, int32_t Hi, int32_t Wi,
                             int32_t C, int8_t *Y, int64_t y_bstride, int32_t Ho, int32_t Wo,
                             ilw_stream_t stream) {
    if (B < 0 || Hi < 1 || Wi < 1 || Ho < 1 || Wo < 1 || C < 16 || C % 16)
        return fail(ILW_ERR_UNSUPPORTED, "resample: bad sizes (C=%d must be a multiple of 16)", C);
    if (B == 0) return ILW_OK;
    if (!X || !Y || !aligned(X, 16) || !aligned(Y, 16) || x_bstride < (int64_t)Hi * Wi || y_bstride < (int64_t)Ho * Wo)
        return fail(ILW_ERR_INVALID_ARG, "resample: NULL, misaligned or overlapping batch strides");
    if (g_check_only) return ILW_OK;
    return cuda_status(ilw::launch_resample(X, x_bstride, B, Hi, Wi, C, Y, y_bstride, Ho, Wo, (cudaStream_t)stream),
                       "resample_nearest");
}

namespace {
struct DecBufs {
    int8_t *qk_in, *v_in, *qkv, *o, *qc, *value, *samp, *fin, *h;
    __half *qkv64;  // heads of dh < 64: q|k|v widened to 64 columns per head (fp16-carried int8)
    int8_t *o64;    // and the attention output at 64 columns per head
    int16_t *x1, *t1, *off16, *att16, *x2, *t2, *x3;
    int32_t *off32, *att32;
    uint8_t *w;
    size_t bytes;
};
DecBufs dec_layout(char *ws, int32_t B, int32_t Q, int64_t S_total, int32_t d, int32_t F, int32_t H, int32_t L,
                   int32_t P) {
    const size_t M = (size_t)B * Q, MS = (size_t)B * S_total, lp = (size_t)H * L * P;
    DecBufs b{};
    size_t off = 0;
    auto take = [&](size_t n) {
        char *p = ws ? ws + off : nullptr;
        off += align256(n);
        return p;
    };
    b.qk_in = (int8_t *)take(M * d);
    b.v_in = (int8_t *)take(M * d);
    b.qkv = (int8_t *)take(M * 3 * d);
    b.o = (int8_t *)take(M * d);
    if (d / H < 64) {
        b.qkv64 = (__half *)take(M * 3 * (size_t)H * 64 * 2);
        b.o64 = (int8_t *)take(M * (size_t)H * 64);
    }
    b.x1 = (int16_t *)take(M * d * 2);
    b.t1 = (int16_t *)take(M * d * 2);
    b.qc = (int8_t *)take(M * d);
    b.value = (int8_t *)take(MS * d);
    b.off16 = (int16_t *)take(M * lp * 2 * 2);
    b.off32 = (int32_t *)take(M * lp * 2 * 4);
    b.att16 = (int16_t *)take(M * lp * 2);
    b.att32 = (int32_t *)take(M * lp * 4);
    b.w = (uint8_t *)take(M * lp);
    b.samp = (int8_t *)take(M * d);
    b.x2 = (int16_t *)take(M * d * 2);
    b.t2 = (int16_t *)take(M * d * 2);
    b.fin = (int8_t *)take(M * d);
    b.h = (int8_t *)take(M * F);
    b.x3 = (int16_t *)take(M * d * 2);
    b.bytes = off;
    return b;
}
}  // namespace

size_t ilwdetr_decoder_workspace_bytes(int32_t B, int32_t Q, int64_t S_total, int32_t d, int32_t F,
                                       int32_t H, int32_t L, int32_t P) {
    if (B < 0 || Q < 0 || S_total < 0 || d < 0 || F < 0 || H < 1 || L < 1 || P < 1) return 0;
    return dec_layout(nullptr, B, Q, S_total, d, F, H, L, P).bytes;
}

int ilwdetr_decoder_layer_forward(const ilw_decoder_params_t *p, const int16_t *tgt, const int16_t *pos,
                                  const int8_t *memory, const int32_t *level_hw, int32_t L,
                                  const int32_t *ref_q16, int32_t B, int32_t Q, int16_t *out,
                                  void *workspace, size_t workspace_bytes, ilw_stream_t stream) {
    if (!p || p->struct_size != sizeof(ilw_decoder_params_t))
        return fail(ILW_ERR_INVALID_ARG, "decoder params NULL or struct_size mismatch");
    const int32_t d = p->d, H = p->H, F = p->F, P = p->P;
    if (d < 16 || d % 16 || H < 1 || d % H || (d / H != 32 && d / H != 64) || F < 16 || F % 16 || P < 1)
        return fail(ILW_ERR_INVALID_ARG, "decoder: d=%d H=%d F=%d P=%d unsupported", d, H, F, P);
    if (L != p->L || L < 1 || L > 8 || !level_hw) return fail(ILW_ERR_INVALID_ARG, "decoder: bad levels");
    if (B < 0 || Q < 0) return fail(ILW_ERR_INVALID_ARG, "decoder: negative sizes");
    if (B == 0 || Q == 0) return ILW_OK;
    if (!tgt || !pos || !memory || !ref_q16 || !out || (const void *)out == (const void *)tgt)
        return fail(ILW_ERR_INVALID_ARG, "decoder: NULL or aliased tensors");
    int64_t S_total = 0;
    for (int l = 0; l < L; ++l) S_total += (int64_t)level_hw[2 * l] * level_hw[2 * l + 1];
    const size_t need = ilwdetr_decoder_workspace_bytes(B, Q, S_total, d, F, H, L, P);
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < need)
        return fail(ILW_ERR_INVALID_ARG, "decoder: workspace NULL, misaligned or smaller than %zu bytes", need);
    const DecBufs b = dec_layout((char *)workspace, B, Q, S_total, d, F, H, L, P);
    const int32_t M = B * Q, LP = L * P, HLP = H * LP;
    const int64_t MS = (int64_t)B * S_total;
    return checked_then_run([&]() -> int {
        int rc;
#define ILW_TRY(x) \
        if ((rc = (x))) return rc
        // self-attention
        ILW_TRY(ilwdetr_requant(tgt, 16, d, M, d, p->m_q1, p->s_q1, pos, d, M, p->m_q2, p->s_q2, 8, b.qk_in, d, stream));
        ILW_TRY(ilwdetr_requant(tgt, 16, d, M, d, p->m_v1, p->s_v1, nullptr, 0, 1, 0, 1, 8, b.v_in, d, stream));
        ILW_TRY(ilwdetr_gemm_requant(b.qk_in, d, p->w_qk, p->b_qk, p->m_qk, p->s_qk, M, 2 * d, d, 8, b.qkv, 3 * d, nullptr,
                                     stream));
        ILW_TRY(ilwdetr_gemm_requant(b.v_in, d, p->w_v, p->b_v, p->m_v, p->s_v, M, d, d, 8, b.qkv + 2 * d, 3 * d, nullptr,
                                     stream));
        if (d / H < 64) {
            // heads of 32 columns run on the tensor-memory attention of 64-column heads: q|k|v widened with
            // zero columns (nothing added to q.k, zero outputs), the output narrowed back
            const int64_t w = (int64_t)H * 64;
            if (!g_check_only) {
                cudaError_t e = ilw::launch_head_pad64(b.qkv, 3 * d, M, 3 * H, d / H, b.qkv64, (cudaStream_t)stream);
                if (e != cudaSuccess) return cuda_status(e, "decoder head pad");
            }
            ILW_TRY(ilwdetr_shiftmax_attn(b.qkv64, b.qkv64 + w, b.qkv64 + 2 * w, 3 * w, ILW_I8_IN_F16, B, Q, H, 64, 0, &p->smx,
                                          p->m_o, p->s_o, b.o64, 8, w, stream));
            if (!g_check_only) {
                cudaError_t e = ilw::launch_head_compact(b.o64, w, M, H, d / H, b.o, d, (cudaStream_t)stream);
                if (e != cudaSuccess) return cuda_status(e, "decoder head compact");
            }
        } else {
            ILW_TRY(ilwdetr_shiftmax_attn(b.qkv, b.qkv + d, b.qkv + 2 * d, 3 * d, 8, B, Q, H, d / H, 0, &p->smx, p->m_o,
                                          p->s_o, b.o, 8, d, stream));
        }
        ilw_residual_t r1{tgt, d, M, p->m_r1, p->s_r1};
        ILW_TRY(ilwdetr_gemm_requant(b.o, d, p->w_o, p->b_o, p->m_oc, p->s_oc, M, d, d, 16, b.x1, d, &r1, stream));
        ILW_TRY(ilwdetr_int_layernorm(b.x1, 16, d, M, d, p->ln1_beta, p->ln1_mult, p->ln1_shift, p->ln_iters, b.t1, 16, d,
                                      stream));
        // deformable cross-attention
        ILW_TRY(ilwdetr_requant(b.t1, 16, d, M, d, p->m_c1, p->s_c1, pos, d, M, p->m_c2, p->s_c2, 8, b.qc, d, stream));
        ILW_TRY(ilwdetr_gemm_requant(memory, d, p->w_val, p->b_val, p->m_val, p->s_val, (int32_t)MS, d, d, 8, b.value, d,
                                     nullptr, stream));
        ILW_TRY(ilwdetr_gemm_requant(b.qc, d, p->w_off, p->b_off, p->m_off, p->s_off, M, 2 * HLP, d, 16, b.off16, 2 * HLP,
                                     nullptr, stream));
        ILW_TRY(ilwdetr_gemm_requant(b.qc, d, p->w_att, p->b_att, p->m_att, p->s_att, M, HLP, d, 16, b.att16, HLP, nullptr,
                                     stream));
        // int16 -> int32 containers (rq with m = 2^30, s = 30 is the identity)
        ILW_TRY(ilwdetr_requant(b.off16, 16, 2 * HLP, M, 2 * HLP, 1 << 30, 30, nullptr, 0, 1, 0, 1, 32, b.off32, 2 * HLP,
                                stream));
        ILW_TRY(ilwdetr_requant(b.att16, 16, HLP, M, HLP, 1 << 30, 30, nullptr, 0, 1, 0, 1, 32, b.att32, HLP, stream));
        ILW_TRY(ilwdetr_shiftmax_rows(b.att32, LP, (int64_t)M * H, LP, &p->smx_w, b.w, LP, stream));
        ILW_TRY(ilwdetr_deform_attn(b.value, level_hw, L, ref_q16, b.off32, b.w, B, Q, H, P, d / H, p->m_s, p->s_s, b.samp,
                                    stream));
        ilw_residual_t r2{b.t1, d, M, p->m_r2, p->s_r2};
        ILW_TRY(ilwdetr_gemm_requant(b.samp, d, p->w_o2, p->b_o2, p->m_o2, p->s_o2, M, d, d, 16, b.x2, d, &r2, stream));
        ILW_TRY(ilwdetr_int_layernorm(b.x2, 16, d, M, d, p->ln2_beta, p->ln2_mult, p->ln2_shift, p->ln_iters, b.t2, 16, d,
                                      stream));
        // FFN
        ILW_TRY(ilwdetr_requant(b.t2, 16, d, M, d, p->m_f, p->s_f, nullptr, 0, 1, 0, 1, 8, b.fin, d, stream));
        ILW_TRY(ilwdetr_gemm_gelu(b.fin, d, p->w_fc1, p->b_fc1, p->m_fc1, p->s_fc1, M, F, d, &p->gelu, p->m_g, p->s_g, b.h,
                                  F, stream));
        ilw_residual_t r3{b.t2, d, M, p->m_r3, p->s_r3};
        ILW_TRY(ilwdetr_gemm_requant(b.h, F, p->w_fc2, p->b_fc2, p->m_fc2, p->s_fc2, M, d, F, 16, b.x3, d, &r3, stream));
        return ilwdetr_int_layernorm(b.x3, 16, d, M, d, p->ln3_beta, p->ln3_mult, p->ln3_shift, p->ln_iters, out, 16, d,
                                     stream);
#undef ILW_TRY
    });
}

// ---------------------------------------------------------------- detection head, two-stage selection
int ilwdetr_int_sigmoid(const int32_t *X, int32_t *Y, int64_t n, const ilw_sigmoid_t *p, ilw_stream_t stream) {
    if (!p) return fail(ILW_ERR_INVALID_ARG, "int_sigmoid: params NULL");
    if (p->I0 < 1 || p->I0 >= (1 << 15)) return fail(ILW_ERR_INVALID_ARG, "int_sigmoid I0=%d outside [1, 2^15)", p->I0);
    if (p->k_inter < 0 || p->k_inter > 16)
        return fail(ILW_ERR_INVALID_ARG, "int_sigmoid k_inter=%d outside [0, 16]", p->k_inter);
    if (((int64_t)p->I0 << (p->k_inter + 1)) >= ((int64_t)1 << 31))
        return fail(ILW_ERR_INVALID_ARG, "int_sigmoid I0 * 2^(k_inter+1) must be < 2^31");
    if (p->k_out < 1 || p->k_out > 24) return fail(ILW_ERR_INVALID_ARG, "int_sigmoid k_out=%d outside [1, 24]", p->k_out);
    if (n < 0) return fail(ILW_ERR_INVALID_ARG, "int_sigmoid: n < 0");
    if (n == 0) return ILW_OK;
    if (!X || !Y || !aligned(X, 16) || !aligned(Y, 16))
        return fail(ILW_ERR_INVALID_ARG, "int_sigmoid: NULL or not 16-byte aligned");
    if (g_check_only) return ILW_OK;
    return cuda_status(ilw::launch_int_sigmoid(X, Y, n, ilw::make_shiftexp(p->I0, p->k_inter), p->k_out,
                                               (cudaStream_t)stream),
                       "int_sigmoid");
}

int ilwdetr_relu_i8(const int8_t *X, int8_t *Y, int64_t n, ilw_stream_t stream) {
    if (n < 0) return fail(ILW_ERR_INVALID_ARG, "relu_i8: n < 0");
    if (n == 0) return ILW_OK;
    if (!X || !Y || !aligned(X, 4) || !aligned(Y, 4)) return fail(ILW_ERR_INVALID_ARG, "relu_i8: NULL or misaligned");
    if (g_check_only) return ILW_OK;
    return cuda_status(ilw::launch_relu_i8(X, Y, n, (cudaStream_t)stream), "relu_i8");
}

int ilwdetr_topk(const int32_t *S, int64_t lds, int32_t rows, int32_t N, int32_t K, int32_t *vals, int32_t *idx,
                 ilw_stream_t stream) {
    if (rows < 0 || N < 1 || K < 1 || K > N || lds < N)
        return fail(ILW_ERR_INVALID_ARG, "topk: bad sizes rows=%d N=%d K=%d", rows, N, K);
    if (N > 16384) return fail(ILW_ERR_UNSUPPORTED, "topk: N=%d above 16384", N);
    if (rows == 0) return ILW_OK;
    if (!S || !vals || !idx || !aligned(S, 4) || !aligned(vals, 4) || !aligned(idx, 4))
        return fail(ILW_ERR_INVALID_ARG, "topk: NULL or misaligned");
    if (g_check_only) return ILW_OK;
    return cuda_status(ilw::launch_topk(S, lds, rows, N, K, vals, idx, (cudaStream_t)stream), "topk");
}

int ilwdetr_gather_rows(const void *src, int64_t src_ld, int64_t src_rows, const int32_t *idx, int64_t n,
                        int64_t row_bytes, void *dst, int64_t dst_ld, ilw_stream_t stream) {
    if (n < 0 || row_bytes < 0 || src_rows < 0 || row_bytes % 4 || src_ld % 4 || dst_ld % 4 || src_ld < row_bytes ||
        dst_ld < row_bytes)
        return fail(ILW_ERR_INVALID_ARG, "gather_rows: bad sizes (row bytes and strides multiples of 4)");
    if (n == 0 || row_bytes == 0) return ILW_OK;
    if (!src || !idx || !dst || !aligned(src, 4) || !aligned(dst, 4) || !aligned(idx, 4))
        return fail(ILW_ERR_INVALID_ARG, "gather_rows: NULL or misaligned");
    if (g_check_only) return ILW_OK;
    return cuda_status(ilw::launch_gather_rows(src, src_ld, src_rows, idx, n, row_bytes, dst, dst_ld, (cudaStream_t)stream),
                       "gather_rows");
}

int ilwdetr_ivit_shiftgelu(const int32_t *X, int64_t ldx, int64_t rows, int32_t L, int32_t *Y, int64_t ldy,
                           const ilw_gelu_t *p, ilw_stream_t stream) {
    int rc = check_gelu(p);
    if (rc) return rc;
    if (rows < 0 || L < 1 || ldx < L || ldy < L) return fail(ILW_ERR_INVALID_ARG, "ivit_shiftgelu: bad sizes");
    if (rows == 0) return ILW_OK;
    if (!X || !Y || !aligned(X, 4) || !aligned(Y, 4)) return fail(ILW_ERR_INVALID_ARG, "ivit_shiftgelu: NULL or misaligned");
    if (g_check_only) return ILW_OK;
    return cuda_status(ilw::launch_ivit_shiftgelu(X, ldx, rows, L, Y, ldy, ilw::make_gelu(*p), (cudaStream_t)stream),
                       "ivit_shiftgelu");
}

}  // extern "C"
