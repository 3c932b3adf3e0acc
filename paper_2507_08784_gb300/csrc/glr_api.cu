// C ABI of libglr.so: handle lifetime and the per-step schedule of Algorithm 3 (Semi-Lazy SVD
// refresh every tau steps, Approx-Top-r selection otherwise), with the host helpers the library's
// other host files share (glr_host.cuh).  All device work is enqueued on the caller's stream; the
// host only tracks the schedule.  The refresh orchestration is in glr_refresh_host.cu, the
// checkpoints and introspection calls in glr_introspect.cu.
#include "glr_host.cuh"

using namespace glr;
using namespace glr::host;

namespace glr {
namespace host {

thread_local std::string g_create_err;
thread_local float* g_ws = nullptr;

int fail(glr_handle* h, int code, const char* fmt, const char* a, int line) {
    char buf[512];
    snprintf(buf, sizeof(buf), fmt, a, line);
    if (h) h->err = buf; else g_create_err = buf;
    return code;
}



cudaEvent_t take_event(glr_handle* h) {
    if (!h->free_events.empty()) {
        cudaEvent_t e = h->free_events.back();
        h->free_events.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
}

void phase_begin(glr_handle* h, int phase, cudaStream_t st) {
    if (!h->prof) return;
    h->cur_phase = phase;
    h->cur_start = take_event(h);
    h->cur_launch0 = h->launches;
    cudaEventRecord(h->cur_start, st);
}

void phase_end(glr_handle* h, cudaStream_t st) {
    if (!h->prof || h->cur_phase < 0) return;
    cudaEvent_t b = take_event(h);
    cudaEventRecord(b, st);
    h->recs.push_back({h->cur_phase, h->cur_start, b, h->launches - h->cur_launch0});
    h->cur_phase = -1;
}



void free_all(glr_handle* h) {
    for (void* p : h->allocs) cudaFree(p);
    h->allocs.clear();
    h->alloc_bytes.clear();
}

// cuTensorMapEncodeTiled from the driver, looked up once through the runtime (no libcuda link).
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            p = nullptr;
        return reinterpret_cast<EncodeTiledFn>(p);
    }();
    return fn;
}

// Row-major (rows x cols) matrices, `depth` of them back to back, read in boxes of 16 columns x
// mma_tma_box_rows(rows) rows; fp32 with the 64-byte swizzle, bf16 with the 32-byte one.
bool encode_strip_map(CUtensorMap* map, const void* base, int rows, int cols, int depth, int gsize) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[3] = {(cuuint64_t)cols, (cuuint64_t)rows, (cuuint64_t)depth};
    const cuuint64_t strides[2] = {(cuuint64_t)cols * gsize, (cuuint64_t)cols * gsize * rows};
    const cuuint32_t box[3] = {16, (cuuint32_t)mma_tma_box_rows(rows), 1};
    const cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, gsize == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, depth > 1 ? 3 : 2,
              const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
              gsize == 2 ? CU_TENSOR_MAP_SWIZZLE_32B : CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_map(CUtensorMap* map, CUtensorMapDataType dtype, const void* base, int rank, const uint64_t* dims,
                const uint64_t* strides, const uint32_t* box, CUtensorMapSwizzle swz) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t d[3], s[2];
    cuuint32_t b[3], e[3] = {1, 1, 1};
    for (int i = 0; i < rank; ++i) { d[i] = dims[i]; b[i] = box[i]; }
    for (int i = 0; i + 1 < rank; ++i) s[i] = strides[i];
    return fn(map, dtype, rank, const_cast<void*>(base), d, s, b, e, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// fp32 operand of the tcgen05 path: `rank` dims (innermost first), byte strides of dims 1..,
// box {32, box[1], 1}, 128-byte swizzle, out-of-range elements read as zero.
bool encode_f32_map(CUtensorMap* map, const float* base, int rank, const uint64_t* dims, const uint64_t* strides,
                    const uint32_t* box) {
    return encode_map(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, base, rank, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_128B);
}

// The descriptor of node i's gradient buffer, re-encoded only when the buffer changes.
bool gradient_map(glr_handle* h, int i, const void* ptr, CUtensorMap* out) {
    glr_handle::GMap* slots = &h->gmaps[2 * (size_t)i];
    for (int q = 0; q < 2; ++q)
        if (slots[q].ptr == ptr) { *out = slots[q].map; return true; }
    slots[1] = slots[0];
    if (!encode_strip_map(&slots[0].map, ptr, h->mp, h->np, 1, (int)h->gsize)) { slots[0].ptr = nullptr; return false; }
    slots[0].ptr = ptr;
    *out = slots[0].map;
    return true;
}


GemmDesc gd(int M, int N, int K, const float* A, int64_t sAi, int64_t sAp, const float* B, int64_t sBp,
            int64_t sBj, float* C, int64_t sCi, int64_t sCj, float alpha, float beta) {
    GemmDesc d{};
    d.ws = g_ws;
    d.ws_floats = g_ws ? kGemmWsFloats : 0;
    d.M = M; d.N = N; d.K = K; d.batch = 1; d.alpha = alpha; d.beta = beta;
    d.A = A; d.sAi = sAi; d.sAp = sAp;
    d.B = B; d.sBp = sBp; d.sBj = sBj;
    d.C = C; d.sCi = sCi; d.sCj = sCj;
    return d;
}

// A plain product C = alpha A B + beta C (GemmDesc semantics) through cuBLAS in its fp32-emulating
// tensor-core mode (CUBLAS_COMPUTE_32F_EMULATED_16BFX9: each fp32 operand split into three bf16
// parts, the partial products accumulated in fp32; fp32-level accuracy).  Returns 1 when the
// strides have no column-major reading (the caller then uses gemm_f32).
int gemm_cublas(glr_handle* h, const GemmDesc& d0, cudaStream_t st) {
    GemmDesc d = d0;
    if (d.sCi != 1) {                       // row-major C: form C^T = B^T A^T instead
        if (d.sCj != 1) return 1;
        GemmDesc t = d;
        t.M = d.N; t.N = d.M;
        t.A = d.B; t.sAi = d.sBj; t.sAp = d.sBp; t.sAz = d.sBz;
        t.B = d.A; t.sBp = d.sAp; t.sBj = d.sAi; t.sBz = d.sAz;
        t.sCi = d.sCj; t.sCj = d.sCi;
        d = t;
    }
    cublasOperation_t ta, tb;
    int64_t lda, ldb;
    if (d.sAi == 1 && d.sAp >= d.M) { ta = CUBLAS_OP_N; lda = d.sAp; }
    else if (d.sAp == 1 && d.sAi >= d.K) { ta = CUBLAS_OP_T; lda = d.sAi; }
    else return 1;
    if (d.sBp == 1 && d.sBj >= d.K) { tb = CUBLAS_OP_N; ldb = d.sBj; }
    else if (d.sBj == 1 && d.sBp >= d.N) { tb = CUBLAS_OP_T; ldb = d.sBp; }
    else return 1;
    const int64_t ldc = d.sCj;
    if (ldc < d.M || lda > INT32_MAX || ldb > INT32_MAX || ldc > INT32_MAX) return 1;
    const int slot = st == h->rstream ? 1 : 0;
    if (!h->cb[slot] && cublasCreate(&h->cb[slot]) != CUBLAS_STATUS_SUCCESS) {
        h->cb[slot] = nullptr;
        return fail(h, GLR_ECUDA, "cublasCreate failed%s");
    }
    if (cublasSetStream(h->cb[slot], st) != CUBLAS_STATUS_SUCCESS) return fail(h, GLR_ECUDA, "cublasSetStream failed%s");
    const float alpha = d.alpha, beta = d.beta;
    const cublasStatus_t cs = cublasGemmStridedBatchedEx(
        h->cb[slot], ta, tb, d.M, d.N, d.K, &alpha, d.A, CUDA_R_32F, (int)lda, d.sAz, d.B, CUDA_R_32F, (int)ldb,
        d.sBz, &beta, d.C, CUDA_R_32F, (int)ldc, d.sCz, d.batch, CUBLAS_COMPUTE_32F_EMULATED_16BFX9, CUBLAS_GEMM_DEFAULT);
    if (cs != CUBLAS_STATUS_SUCCESS)
        return fail(h, GLR_ECUDA, "cuBLAS GEMM failed with status %s", std::to_string(static_cast<int>(cs)).c_str());
    return GLR_OK;
}

// C = alpha A B + beta C: products of at least 2^26 flops through cuBLAS (above), the rest with
// gemm_f32 (k_stream.cu).
int gemm(glr_handle* h, const GemmDesc& d, cudaStream_t st) {
    if (2.0 * d.M * d.N * (double)d.K * d.batch >= 67108864.0) {
        const int rc = gemm_cublas(h, d, st);
        if (rc != 1) return rc;
    }
    GLR_LAUNCH(h, 1, gemm_f32(d, st));
    return GLR_OK;
}

int fail_cuda(glr_handle* h, cudaError_t e, const char* file, int line) {
    const char* base = std::strrchr(file, '/');
    const std::string where = std::string(cudaGetErrorString(e)) + " (" + (base ? base + 1 : file) + ":" +
                              std::to_string(line) + ")";
    return fail(h, GLR_ECUDA, "CUDA error %s", where.c_str());
}

}  // namespace host
}  // namespace glr

namespace {

// Rbar = P^T Mbar; Ghat = P Rbar; optimizer.
int project_and_update(glr_handle* h, float* X, cudaStream_t st) {
    const int mp = h->mp, np = h->np, r = h->r;
    {
        PhaseScope ps(h, GLR_PH_PROJECT, st);
        GLR_GEMM(h, gd(r, np, mp, h->P, 1, r, h->Mbar, np, 1, h->Rbar, np, 1), st);
    }
    PhaseScope ps(h, GLR_PH_UPDATE, st);
    UpdateArgs u{};
    u.mp = mp; u.np = np; u.r = r; u.transposed = h->transposed; u.compressed = 1;
    if (h->tc) {
        // Ghat = P Rbar as a library product written straight into X's layout (transposed when
        // m > n), then one elementwise optimizer pass
        if (h->transposed)
            GLR_GEMM(h, gd(mp, np, r, h->P, r, 1, h->Rbar, np, 1, h->mn_scratch, 1, mp), st);
        else
            GLR_GEMM(h, gd(mp, np, r, h->P, r, 1, h->Rbar, np, 1, h->mn_scratch, np, 1), st);
        u.compressed = 0;
        u.optimizer = h->s.optimizer; u.lr = h->s.lr; u.beta1 = h->s.beta1; u.beta2 = h->s.beta2; u.eps = h->s.eps;
        u.P = h->P; u.Rbar = h->Rbar; u.Mbar = h->mn_scratch; u.X = X; u.Mo = h->Mo; u.Vo = h->Vo;
        GLR_LAUNCH(h, 1, update_streamed_flat(u, st));
        return GLR_OK;
    }
    u.optimizer = h->s.optimizer; u.lr = h->s.lr; u.beta1 = h->s.beta1; u.beta2 = h->s.beta2; u.eps = h->s.eps;
    u.P = h->P; u.Rbar = h->Rbar; u.Mbar = h->Mbar; u.X = X; u.Mo = h->Mo; u.Vo = h->Vo;
    GLR_LAUNCH(h, 1, update(u, st));
    return GLR_OK;
}

int uncompressed_update(glr_handle* h, float* X, cudaStream_t st) {
    UpdateArgs u{};
    u.mp = h->mp; u.np = h->np; u.r = h->r; u.transposed = h->transposed; u.compressed = 0;
    u.optimizer = h->s.optimizer; u.lr = h->s.lr; u.beta1 = h->s.beta1; u.beta2 = h->s.beta2; u.eps = h->s.eps;
    u.P = h->P; u.Rbar = h->Rbar; u.Mbar = h->Mbar; u.X = X; u.Mo = h->Mo; u.Vo = h->Vo;
    GLR_LAUNCH(h, 1, update(u, st));
    return GLR_OK;
}

// The optimizers outside the fused update kernels — the AMSGrad-type step of Appendix A and
// bias-corrected AdamW — with Ghat = Mbar (uncompressed) or P Rbar, both products formed here
// (Rbar = P^T Mbar): one path for every kernel family.
bool separate_optimizer(const glr_handle* h) {
    return h->s.optimizer == GLR_AMSGRAD || h->s.optimizer == GLR_ADAMW || h->s.optimizer == GLR_GALORE_ADAM;
}

// Algorithm 5 (every step compressed with the Lazy-SVD P): the subspace state is zeroed at a
// refresh, advanced with Rbar = P^T Mbar, and X moves by lr P (M / (sqrt(V) + eps)).
int galore_update(glr_handle* h, float* X, bool refresh, cudaStream_t st) {
    const int mp = h->mp, np = h->np, r = h->r;
    const size_t rn = (size_t)r * np;
    {
        PhaseScope ps(h, GLR_PH_PROJECT, st);
        GLR_GEMM(h, gd(r, np, mp, h->P, 1, r, h->Mbar, np, 1, h->Rbar, np, 1), st);
    }
    PhaseScope ps(h, GLR_PH_UPDATE, st);
    if (refresh) {
        GLR_CK(h, cudaMemsetAsync(h->Mo, 0, rn * 4, st));
        GLR_CK(h, cudaMemsetAsync(h->Vo, 0, rn * 4, st));
    }
    GLR_LAUNCH(h, 1, galore_moments(h->Rbar, (int64_t)rn, h->Mo, h->Vo, h->galr, h->s.beta1, h->s.beta2, h->s.eps,
                                    st));
    GLR_GEMM(h, gd(mp, np, r, h->P, r, 1, h->galr, np, 1, h->mn_scratch, np, 1), st);
    GLR_LAUNCH(h, 1, step_apply(h->mn_scratch, mp, np, h->transposed, X, h->s.lr, st));
    return GLR_OK;
}

int separate_optimizer_update(glr_handle* h, float* X, bool compressed, bool refresh, cudaStream_t st) {
    const int mp = h->mp, np = h->np, r = h->r;
    if (h->s.optimizer == GLR_GALORE_ADAM) return galore_update(h, X, refresh, st);
    const float* Gh = h->Mbar;
    if (compressed) {
        PhaseScope ps(h, GLR_PH_PROJECT, st);
        GLR_GEMM(h, gd(r, np, mp, h->P, 1, r, h->Mbar, np, 1, h->Rbar, np, 1), st);
        GLR_GEMM(h, gd(mp, np, r, h->P, r, 1, h->Rbar, np, 1, h->mn_scratch, np, 1), st);
        Gh = h->mn_scratch;
    }
    PhaseScope ps(h, GLR_PH_UPDATE, st);
    if (h->s.optimizer == GLR_ADAMW) {
        const double s = static_cast<double>(h->t + 1);      // this step's optimizer step, 1-based
        const float c1 = static_cast<float>(1.0 / (1.0 - std::pow(static_cast<double>(h->s.beta1), s)));
        const float c2 = static_cast<float>(1.0 / (1.0 - std::pow(static_cast<double>(h->s.beta2), s)));
        GLR_LAUNCH(h, 1, adamw_update(Gh, mp, np, h->transposed, X, h->Mo, h->Vo, h->s.lr, h->s.beta1, h->s.beta2,
                                      h->s.eps, h->s.weight_decay, c1, c2, st));
        return GLR_OK;
    }
    GLR_LAUNCH(h, 3, amsgrad_update(Gh, mp, np, h->transposed, X, h->Mo, h->Vo, h->amsv, h->s.lr, h->s.beta1,
                                    h->s.beta2, h->s.eps, st));
    return GLR_OK;
}

int build_selection_P(glr_handle* h, cudaStream_t st) {
    GLR_LAUNCH(h, 1, build_P(h->exact ? 0 : 1, h->mp, h->r, h->k, h->J, h->U, h->Y, h->Yt, h->dsign, h->P, st));
    return GLR_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

void glr::set_global_error(const char* msg) { g_create_err = msg ? msg : ""; }

extern "C" {

int glr_create(int64_t m, int64_t n, int32_t r, int32_t N, const glr_schedule* s, glr_handle** out) {
    g_create_err.clear();
    if (!out || !s) return fail(nullptr, GLR_EINVAL, "null schedule or output pointer%s");
    *out = nullptr;
    if (m < 1 || n < 1 || m > (1 << 20) || n > (1 << 20))
        return fail(nullptr, GLR_EINVAL, "matrix sizes must be in [1, 2^20]%s");
    const int64_t mp = std::min(m, n), np = std::max(m, n);
    if (mp * np > (int64_t(1) << 31)) return fail(nullptr, GLR_EINVAL, "matrix larger than 2^31 elements%s");
    if (r < 1 || r > mp || r > kMaxRank) return fail(nullptr, GLR_EINVAL, "need 1 <= r <= min(m, n) and r <= 512%s");
    if (N < 1 || N > GLR_MAX_NODES) return fail(nullptr, GLR_EINVAL, "need 1 <= N <= GLR_MAX_NODES%s");
    if (s->tau < 1) return fail(nullptr, GLR_EINVAL, "need tau >= 1%s");
    if (s->selection != GLR_SEL_APPROX && s->selection != GLR_SEL_FIXED)
        return fail(nullptr, GLR_EINVAL, "selection must be GLR_SEL_APPROX or GLR_SEL_FIXED%s");
    if (s->refresh_mode != GLR_ALG3 && s->refresh_mode != GLR_ALG4)
        return fail(nullptr, GLR_EINVAL, "unknown refresh_mode%s");
    if (s->optimizer != GLR_MSGD && s->optimizer != GLR_ADAM && s->optimizer != GLR_AMSGRAD && s->optimizer != GLR_ADAMW &&
        s->optimizer != GLR_GALORE_ADAM)
        return fail(nullptr, GLR_EINVAL, "unknown optimizer%s");
    if (s->optimizer == GLR_GALORE_ADAM && (s->refresh_mode != GLR_ALG4 || s->selection != GLR_SEL_FIXED ||
                                            !s->no_error_feedback || s->compress_start != 0))
        return fail(nullptr, GLR_EINVAL,
                    "GLR_GALORE_ADAM (Algorithm 5) needs refresh_mode GLR_ALG4, selection GLR_SEL_FIXED, "
                    "no_error_feedback 1 and compress_start 0%s");
    if (s->grad_dtype != GLR_F32 && s->grad_dtype != GLR_BF16) return fail(nullptr, GLR_EINVAL, "unknown grad_dtype%s");
    if (s->compress_start < 0) return fail(nullptr, GLR_EINVAL, "need compress_start >= 0%s");
    const int k = (s->basis_rank == 0 || s->basis_rank == mp) ? static_cast<int>(mp) : s->basis_rank;
    const bool exact = k == mp;
    if (!exact && (k < r || k > mp)) return fail(nullptr, GLR_EINVAL, "need r <= basis_rank <= min(m, n)%s");
    if (exact && mp > kMaxFullBasis && !tcl_eligible(mp, np, r, N, k, exact, s))
        return fail(nullptr, GLR_EINVAL,
                    "the full basis above min(m, n) = 1024 needs min(m, n) a multiple of 128 up to 4096, "
                    "max(m, n) a multiple of 8, bf16 gradients, MSGD or Adam, 16 <= r <= 128 (r a multiple of 4) "
                    "and N <= 8; or set basis_rank%s");
    if (!exact && k > kMaxTruncBasis) return fail(nullptr, GLR_EINVAL, "basis_rank above 512 is not supported%s");
    if (!exact && (s->power_iters < 1 || s->power_iters > 64)) return fail(nullptr, GLR_EINVAL, "need 1 <= power_iters <= 64%s");

    glr_handle* h = new glr_handle();
    h->m = m; h->n = n; h->mp = static_cast<int>(mp); h->np = static_cast<int>(np);
    h->transposed = m > n ? 1 : 0; h->r = r; h->N = N; h->k = k; h->exact = exact ? 1 : 0;
    h->s = *s; h->gsize = s->grad_dtype == GLR_BF16 ? 2 : 4;
    h->period_start = s->compress_start;
    h->ntiles = static_cast<int>((np + kLambdaTile - 1) / kLambdaTile);
    // the tcgen05 path (k_tc.cu) takes the matrices it can; the strip kernels the rest
    h->tcl = tcl_eligible(mp, np, r, N, k, exact, s) ? 1 : 0;
    if (!h->tcl) {
        // The fused strip kernels keep a whole m' x BN strip (and P) in shared memory and move
        // rows in 16-byte vectors: they need m' <= 2048, rows of a multiple of 4 elements and
        // room for P.
        const int BN = mp <= 512 ? 32 : mp <= 1024 ? 16 : mp <= 2048 ? 8 : mp <= 4096 ? 4 : 0;
        const int gsz = s->grad_dtype == GLR_BF16 ? 2 : 4;
        const bool rows16 = (np % 4 == 0) && (!h->transposed || mp % 4 == 0);
        const size_t lim = 227 * 1024;
        const bool fits_threads = BN && (int64_t)r * BN / 4 <= kUpdateThreads &&
                                  (int64_t)std::max(r, exact ? 0 : k) * BN / 4 <= kFusedThreads;
        if (BN && rows16 && fits_threads &&
            stream_smem_bytes((int)mp, r, k, BN, gsz, h->transposed, exact ? 0 : 1) <= lim &&
            update_smem_bytes((int)mp, r, BN) <= lim) {
            h->fused = 1;
            h->BN = BN;
            h->nstrips = static_cast<int>((np + BN - 1) / BN);
            if (mma_stream_eligible((int)mp, (int)np, r, k, exact ? 0 : 1, h->transposed, gsz) &&
                (int64_t)r * kMmaStrip / 4 <= kUpdateThreads && update_smem_bytes((int)mp, r, kMmaStrip) <= lim) {
                h->mma = 1;
                h->BN = kMmaStrip;
                h->nstrips = static_cast<int>((np + kMmaStrip - 1) / kMmaStrip);
            }
        }
    }
    cudaGetDevice(&h->device);
    const int rpad_tc = (r + 31) & ~31;
    int rc = GLR_OK;
    const size_t MP = mp, NP = np;
    auto A = [&](auto** p, size_t cnt) { if (rc == GLR_OK) rc = alloc(h, p, cnt); };
    A(&h->B, (size_t)N * MP * NP);
    A(&h->Mbar, MP * NP);
    A(&h->Rw, (size_t)N * (h->tcl ? rpad_tc : r) * NP);
    A(&h->Rbar, (size_t)r * NP);
    A(&h->P, MP * r);
    A(&h->Pprev, MP * r);
    A(&h->J, (size_t)r);
    A(&h->lam, MP);
    A(&h->lam_part, MP * std::max(std::max(h->ntiles, h->nstrips), 4 * ((h->np + 127) / 128)));
    const bool galore = s->optimizer == GLR_GALORE_ADAM;
    A(&h->Mo, galore ? (size_t)r * NP : (size_t)m * n);
    if (s->optimizer != GLR_MSGD) A(&h->Vo, galore ? (size_t)r * NP : (size_t)m * n);
    if (s->optimizer == GLR_AMSGRAD) A(&h->amsv, 2);
    if (galore) A(&h->galr, (size_t)r * NP);
    A(&h->dflags, 8);
    A(&h->gemm_ws, (size_t)kGemmWsFloats);
    // the first path with library products when the rank-r products are large
    h->tc = !h->fused && !h->tcl && mp % 4 == 0 && np % 4 == 0 &&
            2.0 * r * (double)mp * (double)np * N >= 67108864.0 ? 1 : 0;
    if (h->tc || separate_optimizer(h)) A(&h->mn_scratch, MP * NP);
    if ((h->tc || h->tcl) && !exact) A(&h->YtJ, (size_t)r * k);
    if (exact) {
        A(&h->jwork, MP * MP);
        A(&h->jpart, (size_t)2 * kGroupMax * kJacobiMaxGrid);
        A(&h->U, MP * MP); A(&h->Hbuf, MP * MP); A(&h->Vbuf, MP * MP);
        A(&h->evals, MP); A(&h->evals_sorted, MP);
    } else {
        const size_t K = k;
        A(&h->Q, MP * K); A(&h->Qn, MP * K); A(&h->Y, MP * K); A(&h->Yt, MP * K);
        A(&h->T, K * K); A(&h->dsign, K); A(&h->Wbar, K * NP); A(&h->Z, NP * K); A(&h->Zn, NP * K);
        A(&h->Hk, K * K); A(&h->Vk, K * K); A(&h->gram, K * K); A(&h->scratch, K * K);
        A(&h->evals, K); A(&h->evals_sorted, K);
        A(&h->YT, K * transposed_pitch(static_cast<int>(mp)));
        A(&h->YtT, K * transposed_pitch(static_cast<int>(mp)));
        if (h->mma) {
            const size_t frag = ((MP + 7) & ~size_t(7)) * ((K + 7) & ~size_t(7));
            A(&h->YF, frag); A(&h->YtF, frag);
        }
        if (k <= 32 && np % 4 == 0 && !h->tcl) {   // grouped power iteration (k_power.cu), row-major Mbar
            const size_t KM = k <= 16 ? 16 : 32, PC = pow_tile(), CH = pow_chunk();
            const size_t nt = (NP + PC - 1) / PC, nr = (MP + PC - 1) / PC, nn = (NP + CH - 1) / CH;
            A(&h->powpart, nn * KM * MP);
            A(&h->powG, std::max(nt, nr) * KM * KM);
            A(&h->powS, K * K);
            h->pow_ok = 1;
        } else {
            A(&h->jpart, (size_t)2 * kGroupMax * kJacobiMaxGrid);   // the grouped k x k Jacobi (refresh)
        }
    }
    if (rc == GLR_OK && h->tcl) rc = tcl_alloc(h);
    if (rc != GLR_OK) {
        g_create_err = h->err;
        free_all(h);
        delete h;
        return rc;
    }
    // U = I (Algorithm 3 input): dense identity, or Q = I[:, :k], Y = T = 0, d = 1.
    std::vector<float> ones(static_cast<size_t>(mp), 1.f);
    cudaError_t e = cudaSuccess;
    if (exact) {
        e = cudaMemcpy2D(h->U, (MP + 1) * 4, ones.data(), 4, 4, MP, cudaMemcpyHostToDevice);
        if (e == cudaSuccess && h->UT) e = cudaMemcpy2D(h->UT, (MP + 1) * 4, ones.data(), 4, 4, MP, cudaMemcpyHostToDevice);
    }
    else {
        e = cudaMemcpy2D(h->Q, ((size_t)k + 1) * 4, ones.data(), 4, 4, k, cudaMemcpyHostToDevice);
        if (e == cudaSuccess) e = cudaMemcpy(h->dsign, ones.data(), 4 * (size_t)k, cudaMemcpyHostToDevice);
    }
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        g_create_err = std::string("CUDA error during initialisation: ") + cudaGetErrorString(e);
        free_all(h);
        delete h;
        return GLR_ECUDA;
    }
    if (cudaStreamCreateWithFlags(&h->rstream, cudaStreamNonBlocking) != cudaSuccess ||
        cudaEventCreateWithFlags(&h->rfork, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&h->rdone, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&h->rpow, cudaEventDisableTiming) != cudaSuccess) {
        g_create_err = "could not create the refresh stream";
        free_all(h);
        delete h;
        return GLR_ECUDA;
    }
    if (h->mma && mma_stream_tma_eligible((int)mp, (int)np, r, k, exact ? 0 : 1, h->transposed, (int)h->gsize) &&
        encode_strip_map(&h->Bmap, h->B, (int)mp, (int)np, N, 4)) {
        h->tma = 1;
        h->gmaps.assign(2 * (size_t)N, glr_handle::GMap{nullptr, CUtensorMap{}});
    }
    h->iotaJ.resize(r);
    for (int q = 0; q < r; ++q) h->iotaJ[q] = q;
    h->n_state_allocs = h->allocs.size();
    if (h->tcl && (rc = tcl_maps(h)) != GLR_OK) {
        g_create_err = h->err;
        glr_destroy(h);
        return rc;
    }
    *out = h;
    return GLR_OK;
}

int glr_destroy(glr_handle* h) {
    if (!h) return GLR_OK;
    cudaDeviceSynchronize();
    for (auto& rec : h->recs) { cudaEventDestroy(rec.a); cudaEventDestroy(rec.b); }
    for (cudaEvent_t e : h->free_events) cudaEventDestroy(e);
    if (h->rstream) cudaStreamDestroy(h->rstream);
    if (h->rfork) cudaEventDestroy(h->rfork);
    if (h->rdone) cudaEventDestroy(h->rdone);
    if (h->rpow) cudaEventDestroy(h->rpow);
    if (h->cdone) cudaEventDestroy(h->cdone);
    for (cudaEvent_t e : h->sfree) if (e) cudaEventDestroy(e);
    if (h->cstream) cudaStreamDestroy(h->cstream);
    if (h->xready) cudaEventDestroy(h->xready);
    if (h->xdone) cudaEventDestroy(h->xdone);
    if (h->xstream) cudaStreamDestroy(h->xstream);
    for (cublasHandle_t c : h->cb) if (c) cublasDestroy(c);
    free_all(h);
    delete h;
    return GLR_OK;
}

}  // extern "C"

namespace {

struct StepPlan {
    glr_handle* h = nullptr;
    const void* const* G = nullptr;
    float* X = nullptr;
    bool warm = false, refresh = false, forced = false, lam_fused = false, compressed = false;
    bool fixed = false;             // Lazy-SVD selection: J = 0..r-1 (top-r of the last refresh)
    bool stream_update = false;   // K1 writes Wbar and K3 streams X without re-reading Mbar (k_update.cu)
};

int check_step_args(glr_handle* h, const void* const* G, float* X) {
    h->err.clear();
    if (!G || !X) return fail(h, GLR_EINVAL, "null gradient array or X%s");
    if (!aligned16(X)) return fail(h, GLR_EINVAL, "X must be 16-byte aligned%s");
    for (int i = 0; i < h->N; ++i)
        if (!G[i] || !aligned16(G[i]))
            return fail(h, GLR_EINVAL, "gradient %s is null or not 16-byte aligned", std::to_string(i).c_str());
    return GLR_OK;
}

// This step's place in the schedule of Algorithm 3: warm-up (uncompressed), refresh
// ((t - start) mod tau == 0, Semi-Lazy SVD), or a compressed step (Approx-Top-r).
void plan_step(StepPlan& p) {
    glr_handle* h = p.h;
    p.warm = h->t < h->s.compress_start;
    p.refresh = !p.warm && (h->force_refresh || ((h->t - h->period_start) % h->s.tau == 0));
    if (p.refresh && h->force_refresh) h->period_start = h->t;
    h->force_refresh = false;
    p.forced = !p.warm && !p.refresh && h->has_forceJ;
    p.fixed = !p.warm && !p.refresh && !p.forced && h->s.selection == GLR_SEL_FIXED;
    p.lam_fused = h->fused && !h->exact && !p.warm && !p.refresh && !p.forced && !p.fixed;
    p.stream_update = p.lam_fused && h->mma && !separate_optimizer(h) &&
                      update_stream_eligible(h->mp, h->r, h->transposed);
    p.compressed = !p.warm && !(p.refresh && h->s.refresh_mode == GLR_ALG3);
    h->forced_this_step = p.forced;
}

// K1 with the first-path kernels: R_w,i = P_prev^T B_i, then compose.
int compose_unfused(StepPlan& p, cudaStream_t st) {
    glr_handle* h = p.h;
    const int mp = h->mp, np = h->np, r = h->r, N = h->N;
    if (!h->e_zero) {
        PhaseScope ps(h, GLR_PH_PREV_PROJECT, st);
        GemmDesc d = gd(r, np, mp, h->Pprev, 1, r, h->B, np, 1, h->Rw, np, 1);
        d.batch = N; d.sAz = 0; d.sBz = (int64_t)mp * np; d.sCz = (int64_t)r * np;
        GLR_GEMM(h, d, st);
        if (h->tc) {
            // B_i <- E_i = B_i - P_prev R_w,i in place (one batched library product); the
            // compose pass below then only adds G_i
            GemmDesc e = gd(mp, np, r, h->Pprev, r, 1, h->Rw, np, 1, h->B, np, 1, -1.f, 1.f);
            e.batch = N; e.sAz = 0; e.sBz = (int64_t)r * np; e.sCz = (int64_t)mp * np;
            GLR_GEMM(h, e, st);
        }
    }
    PhaseScope ps(h, GLR_PH_COMPOSE, st);
    ComposeArgs ca{};
    for (int i = 0; i < N; ++i) ca.G[i] = p.G[i];
    ca.grad_dtype = h->s.grad_dtype; ca.transposed = h->transposed;
    ca.mp = mp; ca.np = np; ca.N = N; ca.r = h->tc ? 0 : r; ca.e_zero = h->e_zero ? 1 : 0;
    ca.write_B = (p.warm || h->s.no_error_feedback) ? 0 : 1;   // B feeds only the error
    ca.B = h->B; ca.Pprev = h->Pprev; ca.Rw = h->Rw; ca.Mbar = h->Mbar; ca.nonfinite = h->dflags + 3;
    if (h->tc) GLR_LAUNCH(h, 1, compose_streamed(ca, st));
    else GLR_LAUNCH(h, 1, compose(ca, st));
    return GLR_OK;
}

// Work per strip CTA (rows x nodes): larger first so the grouped grid ends evenly.
bool heavier(const StepPlan* a, const StepPlan* b) {
    const int64_t wa = (int64_t)a->h->mp * a->h->N, wb = (int64_t)b->h->mp * b->h->N;
    return wa != wb ? wa > wb : a->h < b->h;
}

// K1 fused and grouped: one launch per (strip width, gradient dtype) bucket and chunk.
int compose_fused(std::vector<StepPlan*>& plans, cudaStream_t st) {
    std::vector<StepPlan*> todo(plans);
    std::stable_sort(todo.begin(), todo.end(), heavier);
    static thread_local TmaMaps maps;      // ~20 KiB: kept off the stack
    while (!todo.empty()) {
        glr_handle* f = todo.front()->h;
        const int BN = f->BN, dt = f->s.grad_dtype, mma = f->mma, tma = f->tma;
        const int gmax = tma ? kTmaGMax : kGroupPtrs;
        StreamGroup g{};
        g.BN = BN; g.grad_dtype = dt; g.err = f->dflags + 2;
        size_t smem = 0;
        std::vector<StepPlan*> rest;
        for (StepPlan* p : todo) {
            glr_handle* h = p->h;
            const int used = g.nmat ? g.mat[g.nmat - 1].g_off + g.mat[g.nmat - 1].N : 0;
            if (h->BN != BN || h->s.grad_dtype != dt || h->mma != mma || h->tma != tma ||
                (mma && mma_stream_nq(h->r) != mma_stream_nq(f->r)) || g.nmat == kGroupMax || used + h->N > gmax) {
                rest.push_back(p);
                continue;
            }
            StreamMat& M = g.mat[g.nmat];
            M.mp = h->mp; M.np = h->np; M.N = h->N; M.r = h->r; M.k = h->k;
            M.transposed = h->transposed; M.e_zero = h->e_zero ? 1 : 0; M.write_B = (p->warm || h->s.no_error_feedback) ? 0 : 1;
            M.lam = p->lam_fused ? 1 : 0;
            M.g_off = used;
            M.strip0 = g.total_strips; M.nstrips = h->nstrips;
            M.B = h->B; M.Pprev = h->Pprev; M.Mbar = h->Mbar;
            M.YT = h->YT; M.YtT = h->YtT; M.YF = h->YF; M.YtF = h->YtF; M.part = h->lam_part;
            M.Wbar = p->stream_update ? h->Wbar : nullptr;
            M.nonfinite = h->dflags + 3;
            M.seed = h->s.seed; M.t = static_cast<uint32_t>(h->t);
            for (int i = 0; i < h->N; ++i) g.G[M.g_off + i] = p->G[i];
            if (tma) {
                maps.B[g.nmat] = h->Bmap;
                for (int i = 0; i < h->N; ++i)
                    if (!gradient_map(h, i, p->G[i], &maps.G[M.g_off + i]))
                        return fail(h, GLR_ECUDA, "could not describe gradient %s for tile copies",
                                    std::to_string(i).c_str());
            }
            g.total_strips += h->nstrips;
            smem = std::max(smem, mma ? mma_stream_smem_bytes(h->mp, h->r, h->k, h->exact ? 0 : 1, (int)h->gsize,
                                                              h->transposed, tma)
                                      : stream_smem_bytes(h->mp, h->r, h->k, BN, (int)h->gsize, h->transposed, M.lam));
            g.nmat++;
        }
        {
            PhaseScope ps(f, GLR_PH_COMPOSE, st);
            GLR_LAUNCH(f, 1, mma ? stream_group_mma(g, tma ? &maps : nullptr, smem, st) : stream_group(g, smem, st));
        }
        todo.swap(rest);
    }
    return GLR_OK;
}

// K3 for compressed steps of a truncated basis, grouped: Rbar from K1's Wbar, then one pass
// over X and the optimizer state.
int update_streamed(std::vector<StepPlan*>& plans, cudaStream_t st) {
    std::vector<StepPlan*> todo(plans);
    std::stable_sort(todo.begin(), todo.end(), heavier);
    while (!todo.empty()) {
        glr_handle* h0 = todo.front()->h;
        UpdStreamGroup g{};
        g.optimizer = h0->s.optimizer;
        g.lr = h0->s.lr; g.beta1 = h0->s.beta1; g.beta2 = h0->s.beta2; g.eps = h0->s.eps;
        std::vector<StepPlan*> rest;
        for (StepPlan* p : todo) {
            glr_handle* h = p->h;
            if (h->s.optimizer != g.optimizer || h->s.lr != g.lr || h->s.beta1 != g.beta1 || h->s.beta2 != g.beta2 ||
                h->s.eps != g.eps || h->transposed != h0->transposed || g.nmat == kGroupMax) {
                rest.push_back(p);
                continue;
            }
            UpdStreamMat& M = g.mat[g.nmat++];
            M.mp = h->mp; M.np = h->np; M.r = h->r; M.k = h->k; M.transposed = h->transposed;
            M.tile0 = g.total_tiles; M.ntiles = update_stream_tiles(h->mp, h->np, h->transposed);
            M.J = h->J; M.dsign = h->dsign; M.Yt = h->Yt; M.Wbar = h->Wbar; M.Mbar = h->Mbar; M.P = h->P;
            M.Rbar = h->Rbar; M.X = p->X; M.Mo = h->Mo; M.Vo = h->Vo;
            g.total_tiles += M.ntiles;
        }
        {
            PhaseScope ps(h0, GLR_PH_UPDATE, st);
            GLR_LAUNCH(h0, 1, update_stream_group(g, st));
        }
        todo.swap(rest);
    }
    return GLR_OK;
}

// K3 fused and grouped.
int update_fused(std::vector<StepPlan*>& plans, cudaStream_t st) {
    std::vector<StepPlan*> todo(plans);
    std::stable_sort(todo.begin(), todo.end(), heavier);
    while (!todo.empty()) {
        glr_handle* h0 = todo.front()->h;
        const int BN = h0->BN;
        UpdateGroup g{};
        g.BN = BN; g.optimizer = h0->s.optimizer;
        g.lr = h0->s.lr; g.beta1 = h0->s.beta1; g.beta2 = h0->s.beta2; g.eps = h0->s.eps;
        size_t smem = 0;
        std::vector<StepPlan*> rest;
        for (StepPlan* p : todo) {
            glr_handle* h = p->h;
            if (h->BN != BN || h->s.optimizer != g.optimizer || h->s.lr != g.lr || h->s.beta1 != g.beta1 ||
                h->s.beta2 != g.beta2 || h->s.eps != g.eps || g.nmat == kGroupMax) {
                rest.push_back(p);
                continue;
            }
            UpdateMat& M = g.mat[g.nmat];
            M.mp = h->mp; M.np = h->np; M.r = h->r; M.transposed = h->transposed; M.compressed = p->compressed ? 1 : 0;
            M.strip0 = g.total_strips; M.nstrips = h->nstrips;
            M.P = h->P; M.Rbar = h->Rbar; M.Mbar = h->Mbar; M.X = p->X; M.Mo = h->Mo; M.Vo = h->Vo;
            g.total_strips += h->nstrips;
            smem = std::max(smem, update_smem_bytes(h->mp, h->r, BN));
            g.nmat++;
        }
        {
            PhaseScope ps(h0, GLR_PH_UPDATE, st);
            GLR_LAUNCH(h0, 1, update_group(g, smem, st));
        }
        todo.swap(rest);
    }
    return GLR_OK;
}

// ---- the tcgen05 path (k_tc.cu) -------------------------------------------------------------
// Every op is one grouped launch over the matrices that take part in it (kTcGroupMax per launch).
tc::TcMat tc_mat(const glr_handle* h) {
    tc::TcMat M{};
    M.mp = h->mp; M.np = h->np; M.N = h->N; M.r = h->r; M.rpad = h->rpad; M.k = h->k; M.kpad = h->kpad;
    M.transposed = h->transposed; M.gdtype = h->s.grad_dtype;
    M.seed = h->s.seed; M.t = static_cast<uint32_t>(h->t);
    return M;
}
inline int cdiv(int a, int b) { return (a + b - 1) / b; }

// fill(plan, M, g, first) describes the plan's matrix for the op: 1 = take it, 0 = the plan has
// no part in this op, -1 = it needs another launch (its optimizer settings differ), -2 = failure
// (recorded on the plan's handle).
template <class Fill>
int tc_run(std::vector<StepPlan*> plans, int phase, cudaError_t (*launch)(tc::TcGroup&, cudaStream_t), cudaStream_t st,
           Fill fill) {
    static thread_local tc::TcGroup g;
    while (!plans.empty()) {
        g.nmat = 0; g.total_tiles = 0; g.err = nullptr;
        int gptrs = 0;
        glr_handle* h0 = nullptr;
        std::vector<StepPlan*> rest;
        for (StepPlan* p : plans) {
            glr_handle* h = p->h;
            if (g.nmat == tc::kTcGroupMax || gptrs + h->N > tc::kTcGPtrs) { rest.push_back(p); continue; }
            tc::TcMat M = tc_mat(h);
            const int take = fill(*p, M, g, h0 == nullptr);
            if (take == -2) return GLR_ECUDA;         // the fill recorded the failure on h
            if (take == 0) continue;
            if (take < 0) { rest.push_back(p); continue; }
            if (!h0) { h0 = h; g.err = h->dflags + 2; }
            M.tile0 = g.total_tiles;
            g.total_tiles += M.ntiles;
            M.g_off = gptrs;
            for (int i = 0; i < h->N; ++i) g.G[gptrs + i] = p->G[i];
            gptrs += h->N;
            g.mat[g.nmat++] = M;
        }
        if (h0 && g.total_tiles > 0) {
            PhaseScope ps(h0, phase, st);
            GLR_LAUNCH(h0, 1, launch(g, st));
        }
        plans.swap(rest);
    }
    return GLR_OK;
}

bool tc_needs_lambda(const StepPlan& p) { return p.compressed && !p.refresh && !p.forced && !p.fixed; }

// K1: R_w,i^T = (P_prev^T B_i)^T for matrices with a live error, then the compose pass.
int tcl_compose(std::vector<StepPlan*>& plans, cudaStream_t st) {
    int rc = tc_run(plans, GLR_PH_PREV_PROJECT, tc::launch_prevproj, st, [](StepPlan& p, tc::TcMat& M, tc::TcGroup&, bool) {
        glr_handle* h = p.h;
        if (h->e_zero) return 0;
        M.na = h->tc_na; M.ng = h->tc_ng; M.tn = cdiv(h->np, 128); M.ntiles = M.tn * M.ng;
        M.mA = tcl_map(h, kMapBt); M.mB = tcl_map_PT(h, h->Pprev); M.Rw = h->Rw;
        return 1;
    });
    if (rc != GLR_OK) return rc;
    return tc_run(plans, GLR_PH_COMPOSE, tc::launch_compose, st, [st](StepPlan& p, tc::TcMat& M, tc::TcGroup&, bool) {
        glr_handle* h = p.h;
        M.e_zero = h->e_zero ? 1 : 0;
        M.write_B = (p.warm || h->s.no_error_feedback) ? 0 : 1;
        M.tm = cdiv(h->mp, 128); M.tn = cdiv(h->np, tc::compose_bn()); M.ntiles = M.tm * M.tn;
        M.mA = tcl_map_P(h, h->Pprev); M.mB = tcl_map(h, kMapRwT);
        int rc = GLR_OK;
        M.mD0 = tcl_map(h, kMapBtD);
        M.mD1 = tcl_grad_maps(h, p.G, st, &rc);
        if (rc != GLR_OK) return -2;
        M.B = h->B; M.Mbar = h->Mbar; M.nonfinite = h->dflags + 3;
        M.MbarRow = (p.refresh && h->k <= 256) ? h->Mrow : nullptr;   // the refresh's Mbar Z products
        return 1;
    });
}

auto tc_wbar_fill(bool lam_plans) {
    return [lam_plans](StepPlan& p, tc::TcMat& M, tc::TcGroup&, bool) {
        glr_handle* h = p.h;
        if (!p.compressed || h->exact || tc_needs_lambda(p) != lam_plans) return 0;
        M.ntiles = cdiv(h->np, 256);
        M.mA = tcl_map(h, kMapMbarT); M.mB = tcl_map(h, kMapYT); M.W = h->WT;
        return 1;
    };
}

// Approx-Top-r partials for the matrices that select this step: W = Y^T Mbar, then the scores.
int tcl_lambda(std::vector<StepPlan*>& plans, cudaStream_t st) {
    int rc = tc_run(plans, GLR_PH_LAMBDA, tc::launch_wbar, st, tc_wbar_fill(true));
    if (rc != GLR_OK) return rc;
    rc = tc_run(plans, GLR_PH_LAMBDA, tc::launch_lambda, st, [](StepPlan& p, tc::TcMat& M, tc::TcGroup&, bool) {
        glr_handle* h = p.h;
        if (!tc_needs_lambda(p) || h->exact) return 0;
        M.tm = cdiv(h->mp, 128); M.tn = cdiv(h->np, 128); M.ntiles = M.tm * M.tn;
        M.mA = tcl_map(h, kMapYt); M.mB = tcl_map(h, kMapWT); M.mD0 = tcl_map(h, kMapMbarL);
        M.Mbar = h->Mbar; M.part = h->lam_part;
        return 1;
    });
    if (rc != GLR_OK) return rc;
    // the full basis: the dense scores U^T Mbar with v_j in the epilogue
    return tc_run(plans, GLR_PH_LAMBDA, tc::launch_lambda_u, st, [](StepPlan& p, tc::TcMat& M, tc::TcGroup&, bool) {
        glr_handle* h = p.h;
        if (!tc_needs_lambda(p) || !h->exact) return 0;
        M.tm = cdiv(h->mp, 128); M.tn = cdiv(h->np, 256); M.ntiles = M.tm * M.tn;
        M.mA = tcl_map(h, kMapUT); M.mB = tcl_map(h, kMapMbarT); M.part = h->lam_part;
        return 1;
    });
}

// After J: W for the matrices that did not select (a supplied J, or the refresh of Algorithm 4),
// P = U[:, J] (and P^T), Rbar, then the update pass for every matrix.
int tcl_project(std::vector<StepPlan*>& plans, cudaStream_t st) {
    int rc = tc_run(plans, GLR_PH_PROJECT, tc::launch_wbar, st, tc_wbar_fill(false));
    if (rc != GLR_OK) return rc;
    // YtJ = Yt[J, :] was gathered by the selection launch
    for (StepPlan* p : plans) {                 // a full basis: P = U[:, J] and P^T, gathered
        glr_handle* h = p->h;
        if (!p->compressed || !h->exact) continue;
        PhaseScope ps(h, GLR_PH_SELECT, st);
        GLR_LAUNCH(h, 1, tc::gather_p(h->U, h->mp, h->J, h->r, h->P, tcl_PT_of(h, h->P), st));
    }
    rc = tc_run(plans, GLR_PH_SELECT, tc::launch_pbuild, st, [](StepPlan& p, tc::TcMat& M, tc::TcGroup&, bool) {
        glr_handle* h = p.h;
        if (!p.compressed || h->exact) return 0;
        M.ntiles = cdiv(h->mp, 128);
        M.mA = tcl_map(h, kMapY); M.mB = tcl_map(h, kMapYtJn);
        M.J = h->J; M.dsign = h->dsign; M.Pout = h->P; M.PT = tcl_PT_of(h, h->P);
        return 1;
    });
    if (rc != GLR_OK) return rc;
    // a full basis: Rbar^T = (P^T Mbar)^T by the R_w product on Mbar as a single node
    rc = tc_run(plans, GLR_PH_PROJECT, tc::launch_prevproj, st, [](StepPlan& p, tc::TcMat& M, tc::TcGroup&, bool) {
        glr_handle* h = p.h;
        if (!p.compressed || !h->exact) return 0;
        M.N = 1; M.na = 1; M.ng = 1; M.tn = cdiv(h->np, 128); M.ntiles = M.tn;
        M.mA = tcl_map(h, kMapMbar3); M.mB = tcl_map_PT(h, h->P); M.Rw = h->RbarT;
        return 1;
    });
    if (rc != GLR_OK) return rc;
    rc = tc_run(plans, GLR_PH_PROJECT, tc::launch_rbar, st, [](StepPlan& p, tc::TcMat& M, tc::TcGroup&, bool) {
        glr_handle* h = p.h;
        if (!p.compressed || h->exact) return 0;
        M.ntiles = cdiv(h->np, 128);
        M.mA = tcl_map(h, kMapYtJm); M.mB = tcl_map(h, kMapWT);
        M.J = h->J; M.dsign = h->dsign; M.Mbar = h->Mbar; M.Rbar = h->Rbar; M.RbarT = h->RbarT;
        return 1;
    });
    return rc;
}

// The update pass (K3) of every matrix.
int tcl_update(std::vector<StepPlan*>& plans, cudaStream_t st) {
    return tc_run(plans, GLR_PH_UPDATE, tc::launch_update, st, [st](StepPlan& p, tc::TcMat& M, tc::TcGroup& g, bool first) {
        glr_handle* h = p.h;
        const glr_schedule& s = h->s;
        if (first) {
            g.optimizer = s.optimizer; g.lr = s.lr; g.beta1 = s.beta1; g.beta2 = s.beta2; g.eps = s.eps;
        } else if (g.optimizer != s.optimizer || g.lr != s.lr || g.beta1 != s.beta1 || g.beta2 != s.beta2 ||
                   g.eps != s.eps) {
            return -1;
        }
        M.compressed = p.compressed ? 1 : 0;
        M.tm = cdiv(h->mp, 128); M.tn = cdiv(h->np, 128); M.ntiles = M.tm * M.tn;
        M.mA = tcl_map_P(h, h->P); M.mB = tcl_map(h, kMapRbarT);
        int rc = GLR_OK;
        M.mD0 = tcl_x_map(h, p.X, st, &rc);
        if (rc != GLR_OK) return -2;
        M.mD1 = tcl_map(h, kMapMo); M.mD2 = tcl_map(h, kMapVo); M.mD3 = tcl_map(h, kMapMbarU);
        M.Mbar = h->Mbar; M.X = p.X; M.Mo = h->Mo; M.Vo = h->Vo;
        return 1;
    });
}

int tcl_project_update(std::vector<StepPlan*>& plans, cudaStream_t st) {
    const int rc = tcl_project(plans, st);
    return rc != GLR_OK ? rc : tcl_update(plans, st);
}

// Between K1 and K3: refresh, or Approx-Top-r selection and P.
int select_phase(StepPlan& p, cudaStream_t st) {
    glr_handle* h = p.h;
    const int mp = h->mp, np = h->np, r = h->r;
    int rc = GLR_OK;
    if (p.warm) return GLR_OK;
    if (p.refresh) {
        h->refreshes++;
        h->comm += (int64_t)mp * np;
        if (h->s.refresh_mode == GLR_ALG3) return GLR_OK;
        GLR_CK(h, cudaMemcpyAsync(h->J, h->iotaJ.data(), sizeof(int32_t) * r, cudaMemcpyHostToDevice, st));
        h->comm += (int64_t)r * np;
    } else if (p.fixed) {
        GLR_CK(h, cudaMemcpyAsync(h->J, h->iotaJ.data(), sizeof(int32_t) * r, cudaMemcpyHostToDevice, st));
        h->comm += (int64_t)r * np;
    } else if (p.forced) {
        GLR_CK(h, cudaMemcpyAsync(h->J, h->forceJ.data(), sizeof(int32_t) * r, cudaMemcpyHostToDevice, st));
        h->has_forceJ = false;
        h->comm += (int64_t)r * np + mp;
    } else if (h->tcl) {
        h->comm += (int64_t)r * np + mp;           // the scores come from tcl_lambda
    } else if (!p.lam_fused) {
        PhaseScope ps(h, GLR_PH_LAMBDA, st);
        LambdaArgs la{};
        la.mp = mp; la.np = np; la.seed = h->s.seed; la.t = static_cast<uint32_t>(h->t);
        la.part = h->lam_part; la.ntiles = h->ntiles;
        if (h->exact) {
            la.mode = 0; la.K = mp; la.A = h->U; la.Bm = h->Mbar; la.Mbar = h->Mbar;
        } else {
            const int k = h->k;
            GLR_GEMM(h, gd(k, np, mp, h->Y, 1, k, h->Mbar, np, 1, h->Wbar, np, 1), st);  // Wbar = Y^T Mbar
            la.mode = 1; la.K = k; la.A = h->Yt; la.Bm = h->Wbar; la.Mbar = h->Mbar;
            if (h->tc) {
                // Yt Wbar as a library product into the scratch; the score kernel then forms the
                // row sums of (Mbar - scratch) against v_j (K = 0)
                GLR_GEMM(h, gd(mp, np, k, h->Yt, k, 1, h->Wbar, np, 1, h->mn_scratch, np, 1), st);
                la.K = 0; la.Csub = h->mn_scratch;
            }
        }
        GLR_LAUNCH(h, 1, lambda_partials(la, st));
        h->comm += (int64_t)r * np + mp;
    } else {
        h->comm += (int64_t)r * np + mp;
    }
    return GLR_OK;
}

// arg-top-r (unless J was supplied) and P = U[:, J] for every compressed matrix, grouped.
int select_P_grouped(std::vector<StepPlan>& plans, cudaStream_t st, int stages = 3) {
    SelectGroup g{};
    glr_handle* h0 = nullptr;
    auto flush = [&]() -> int {
        if (g.nmat == 0) return GLR_OK;
        PhaseScope ps(h0, GLR_PH_SELECT, st);
        GLR_LAUNCH(h0, (stages & 1) + 2 * ((stages >> 1) & 1), select_group(g, st, stages));
        g = SelectGroup{};
        h0 = nullptr;
        return GLR_OK;
    };
    for (StepPlan& p : plans) {
        if (!p.compressed) continue;
        glr_handle* h = p.h;
        if (!h0) h0 = h;
        SelectMat& M = g.mat[g.nmat++];
        M.part = h->lam_part;
        M.ntiles = h->tcl ? (h->exact ? 4 * cdiv(h->np, 256) : h->tc_lam_tiles) : p.lam_fused ? h->nstrips : h->ntiles;
        M.mp = h->mp; M.r = h->r; M.k = h->k; M.mode = h->exact ? 0 : 1;
        M.do_select = (!p.refresh && !p.forced && !p.fixed) ? 1 : 0;
        M.dsign = h->exact ? nullptr : h->dsign; M.lam = h->lam; M.J = h->J;
        M.U = h->U; M.Y = h->Y; M.Yt = h->Yt; M.P = h->P;
        M.rbar = p.stream_update ? 1 : 0; M.np = h->np;
        M.Mbar = h->Mbar; M.Wbar = h->Wbar; M.Rbar = h->Rbar;
        M.build_p = (h->tcl || (h->tc && !h->exact)) ? 0 : 1;   // the tcgen05 path builds its own P
        M.YtJ = (h->tcl && !h->exact) ? h->YtJ : nullptr;
        M.out0 = g.total_out;
        g.total_out += (M.build_p ? (int64_t)h->mp * h->r : 0) + (M.rbar ? (int64_t)h->r * h->np : 0);
        if (g.nmat == kGroupMax) {
            int rc = flush();
            if (rc != GLR_OK) return rc;
        }
    }
    int rc = flush();
    if (rc != GLR_OK) return rc;
    if (!(stages & 2)) return GLR_OK;
    // P = U[:, J] of a truncated basis with large products: (E_J - Y Yt[J, :]^T) D_J
    for (StepPlan& p : plans) {
        glr_handle* h = p.h;
        if (!p.compressed || !h->tc || h->exact) continue;
        PhaseScope ps(h, GLR_PH_SELECT, st);
        const int mp = h->mp, r = h->r, k = h->k;
        GLR_LAUNCH(h, 1, wy_columns_gather(h->Yt, h->J, r, k, h->YtJ, st));
        GLR_GEMM(h, gd(mp, r, k, h->Y, k, 1, h->YtJ, 1, k, h->P, r, 1, -1.f, 0.f), st);
        GLR_LAUNCH(h, 1, wy_columns_fix(h->P, h->J, h->dsign, mp, r, k, st));
    }
    return GLR_OK;
}

int update_unfused(StepPlan& p, cudaStream_t st) {
    if (!p.compressed) {
        PhaseScope ps(p.h, GLR_PH_UPDATE, st);
        return uncompressed_update(p.h, p.X, st);
    }
    return project_and_update(p.h, p.X, st);
}

void finish_step(StepPlan& p) {
    glr_handle* h = p.h;
    if (p.warm) {
        h->comm += (int64_t)h->mp * h->np;
        h->last_uncompressed = true;
    } else if (!p.compressed) {
        h->e_zero = true;
        h->last_uncompressed = true;
        h->has_forceJ = false;
    } else {
        std::swap(h->P, h->Pprev);      // Pprev now holds this step's P (deferred E_i = B_i - P P^T B_i)
        h->e_zero = h->s.no_error_feedback != 0;   // without error feedback E_i stays 0
        h->last_uncompressed = false;
    }
    h->t++;
}

int step_group(std::vector<StepPlan>& plans, cudaStream_t st) {
    std::vector<StepPlan*> fused, unfused, tcl;
    for (StepPlan& p : plans) {
        plan_step(p);
        (p.h->tcl ? tcl : p.h->fused ? fused : unfused).push_back(&p);
    }
    int rc;
    if (!fused.empty() && (rc = compose_fused(fused, st)) != GLR_OK) return rc;
    if (!tcl.empty() && (rc = tcl_compose(tcl, st)) != GLR_OK) return rc;
    for (StepPlan* p : unfused)
        if ((rc = compose_unfused(*p, st)) != GLR_OK) return rc;
    // Refreshes (Semi-Lazy SVD) of different matrices are independent: each runs on its
    // handle's side stream after the compose pass, overlapping the others and the selection
    // work of the non-refreshing matrices; the main stream joins them before P is built.
    std::vector<glr_handle*> refreshing, grouped, exact, trunc, tclr;
    for (StepPlan& p : plans) {
        if (!p.refresh) continue;
        glr_handle* h = p.h;
        GLR_CK(h, cudaEventRecord(h->rfork, st));
        GLR_CK(h, cudaStreamWaitEvent(h->rstream, h->rfork, 0));
        refreshing.push_back(h);
        (h->pow_ok ? grouped : h->exact ? exact : (h->tcl && h->k <= 256) ? tclr : trunc).push_back(h);
    }
    if (!grouped.empty() && (rc = refresh_grouped(grouped)) != GLR_OK) return rc;
    if (!exact.empty() && (rc = refresh_exact_grouped(exact)) != GLR_OK) return rc;
    if (!trunc.empty() && (rc = refresh_trunc_grouped(trunc)) != GLR_OK) return rc;
    if (!tclr.empty() && (rc = refresh_tcl_grouped(tclr)) != GLR_OK) return rc;
    for (glr_handle* h : refreshing) GLR_CK(h, cudaEventRecord(h->rdone, h->rstream));
    for (StepPlan& p : plans)
        if ((rc = select_phase(p, st)) != GLR_OK) return rc;
    if (!tcl.empty() && (rc = tcl_lambda(tcl, st)) != GLR_OK) return rc;
    for (glr_handle* h : refreshing) GLR_CK(h, cudaStreamWaitEvent(st, h->rdone, 0));
    if ((rc = select_P_grouped(plans, st)) != GLR_OK) return rc;
    // X is written from here on: a read-back of the previous step's X (glr_step_group_host) ends first
    for (StepPlan& p : plans)
        if (p.h->x_pending) {
            GLR_CK(p.h, cudaStreamWaitEvent(st, p.h->xdone, 0));
            p.h->x_pending = false;
        }
    if (!tcl.empty() && (rc = tcl_project_update(tcl, st)) != GLR_OK) return rc;
    std::vector<StepPlan*> streamed, strips;
    for (StepPlan* p : fused) {
        if (separate_optimizer(p->h)) continue;
        (p->stream_update ? streamed : strips).push_back(p);
    }
    if (!streamed.empty() && (rc = update_streamed(streamed, st)) != GLR_OK) return rc;
    if (!strips.empty() && (rc = update_fused(strips, st)) != GLR_OK) return rc;
    for (StepPlan* p : unfused)
        if (!separate_optimizer(p->h) && (rc = update_unfused(*p, st)) != GLR_OK) return rc;
    for (StepPlan& p : plans)
        if (separate_optimizer(p.h) && (rc = separate_optimizer_update(p.h, p.X, p.compressed, p.refresh, st)) != GLR_OK)
            return rc;
    for (StepPlan& p : plans) finish_step(p);
    return GLR_OK;
}

// ---- data-parallel steps across processes (glr_dp_*) ------------------------------------------
enum : int { kDpWarm = 1, kDpRefresh = 2, kDpForced = 4, kDpFixed = 8, kDpCompressed = 16 };

StepPlan dp_plan(glr_handle* h) {
    StepPlan p;
    p.h = h; p.G = h->dp_G; p.X = nullptr;
    p.warm = h->dp_flags & kDpWarm; p.refresh = h->dp_flags & kDpRefresh; p.forced = h->dp_flags & kDpForced;
    p.fixed = h->dp_flags & kDpFixed; p.compressed = h->dp_flags & kDpCompressed;
    return p;
}

void dp_expose(glr_dp_exchange* ex, float* ptr, int64_t floats) {
    ex->ptr[ex->count] = ptr;
    ex->floats[ex->count] = floats;
    ex->count++;
}

int dp_begin(glr_handle* h, const void* const* G, cudaStream_t st, glr_dp_exchange* ex) {
    for (int i = 0; i < h->N; ++i) h->dp_G[i] = G[i];
    std::vector<StepPlan> plans(1);
    StepPlan& p = plans[0];
    p.h = h; p.G = h->dp_G;
    plan_step(p);
    h->dp_flags = (p.warm ? kDpWarm : 0) | (p.refresh ? kDpRefresh : 0) | (p.forced ? kDpForced : 0) |
                  (p.fixed ? kDpFixed : 0) | (p.compressed ? kDpCompressed : 0);
    std::vector<StepPlan*> v{&p};
    int rc = tcl_compose(v, st);
    if (rc != GLR_OK) return rc;
    if (p.warm || p.refresh) {                 // the node mean: the refresh's input, or Ghat
        dp_expose(ex, h->Mbar, (int64_t)h->mp * h->np);
        return GLR_OK;
    }
    if ((rc = select_phase(p, st)) != GLR_OK) return rc;     // J of a forced / fixed selection
    if (tc_needs_lambda(p)) {                  // this shard's lambda-bar (linear in Mbar)
        if ((rc = tcl_lambda(v, st)) != GLR_OK) return rc;
        if ((rc = select_P_grouped(plans, st, 1)) != GLR_OK) return rc;
        dp_expose(ex, h->lam, h->mp);
    }
    return GLR_OK;
}

int dp_select(glr_handle* h, cudaStream_t st, glr_dp_exchange* ex) {
    std::vector<StepPlan> plans(1, dp_plan(h));
    StepPlan& p = plans[0];
    std::vector<StepPlan*> v{&p};
    int rc;
    if (p.refresh) {                           // the Semi-Lazy SVD of the averaged node mean
        if (h->k <= 256)
            GLR_LAUNCH(h, 1, transpose_pad(h->Mrow, h->np, h->Mbar, h->np, h->mp, st));   // its row-major copy
        GLR_CK(h, cudaEventRecord(h->rfork, st));
        GLR_CK(h, cudaStreamWaitEvent(h->rstream, h->rfork, 0));
        std::vector<glr_handle*> hs{h};
        rc = h->exact ? refresh_exact_grouped(hs) : h->k <= 256 ? refresh_tcl_grouped(hs) : refresh_trunc_grouped(hs);
        if (rc != GLR_OK) return rc;
        GLR_CK(h, cudaEventRecord(h->rdone, h->rstream));
        GLR_CK(h, cudaStreamWaitEvent(st, h->rdone, 0));
        if ((rc = select_phase(p, st)) != GLR_OK) return rc;
    }
    if (!p.compressed) return GLR_OK;          // Ghat = Mbar: nothing more to average
    if ((rc = select_P_grouped(plans, st, 2)) != GLR_OK) return rc;   // lambda-bar came from glr_dp_begin
    if ((rc = tcl_project(v, st)) != GLR_OK) return rc;
    dp_expose(ex, h->RbarT, (int64_t)h->np * h->rpad);       // this shard's Rbar (as Rbar^T)
    return GLR_OK;
}

int dp_finish(glr_handle* h, float* X, cudaStream_t st) {
    std::vector<StepPlan> plans(1, dp_plan(h));
    StepPlan& p = plans[0];
    p.X = X;
    std::vector<StepPlan*> v{&p};
    if (h->x_pending) {                        // a host read-back of X still in flight
        GLR_CK(h, cudaStreamWaitEvent(st, h->xdone, 0));
        h->x_pending = false;
    }
    const int rc = tcl_update(v, st);
    if (rc != GLR_OK) return rc;
    finish_step(p);
    return GLR_OK;
}

}  // namespace

extern "C" {

int glr_step(glr_handle* h, const void* const* G, float* X, void* stream) {
    if (!h) return GLR_EINVAL;
    int rc = check_step_args(h, G, X);
    if (rc != GLR_OK) return rc;
    std::vector<StepPlan> plans(1);
    plans[0].h = h; plans[0].G = G; plans[0].X = X;
    return step_group(plans, static_cast<cudaStream_t>(stream));
}

int glr_step_group(glr_handle* const* handles, int32_t count, const void* const* const* G, float* const* X,
                   void* stream) {
    if (!handles || count < 1 || !G || !X) return fail(nullptr, GLR_EINVAL, "null arrays or count < 1%s");
    std::vector<StepPlan> plans(count);
    for (int j = 0; j < count; ++j) {
        glr_handle* h = handles[j];
        if (!h) return fail(nullptr, GLR_EINVAL, "null handle in the group%s");
        for (int l = 0; l < j; ++l)
            if (handles[l] == h) return fail(nullptr, GLR_EINVAL, "a handle appears twice in the group%s");
        int rc = check_step_args(h, G[j], X[j]);
        if (rc != GLR_OK) return rc;
        plans[j].h = h; plans[j].G = G[j]; plans[j].X = X[j];
    }
    return step_group(plans, static_cast<cudaStream_t>(stream));
}

int glr_step_host(glr_handle* h, const void* const* G_host, float* X, float* X_host_out, void* stream) {
    if (!h) return GLR_EINVAL;
    if (!G_host || !X) return fail(h, GLR_EINVAL, "null gradient array or X%s");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const size_t bytes = static_cast<size_t>(h->m) * h->n * h->gsize;
    if (!h->Gstage) {
        char* p = nullptr;
        int rc = alloc(h, &p, bytes * h->N);
        if (rc != GLR_OK) return rc;
        h->Gstage = p;
        GLR_CK(h, cudaDeviceSynchronize());      // alloc's zero fill is on the legacy stream
    }
    const void* Gd[GLR_MAX_NODES];
    for (int i = 0; i < h->N; ++i) {
        if (!G_host[i]) return fail(h, GLR_EINVAL, "host gradient %s is null", std::to_string(i).c_str());
        char* dst = static_cast<char*>(h->Gstage) + bytes * i;
        GLR_CK(h, cudaMemcpyAsync(dst, G_host[i], bytes, cudaMemcpyHostToDevice, st));
        Gd[i] = dst;
    }
    int rc = glr_step(h, Gd, X, stream);
    if (rc != GLR_OK) return rc;
    if (X_host_out) {
        GLR_CK(h, cudaMemcpyAsync(X_host_out, X, sizeof(float) * h->m * h->n, cudaMemcpyDeviceToHost, st));
        GLR_CK(h, cudaStreamSynchronize(st));
    }
    return GLR_OK;
}

int glr_dp_begin(glr_handle* h, const void* const* G, void* stream, glr_dp_exchange* out) {
    if (!h || !out) return fail(h, GLR_EINVAL, "null handle or exchange descriptor%s");
    h->err.clear();
    *out = glr_dp_exchange{};
    if (!h->tcl) return fail(h, GLR_EINVAL, "data-parallel steps need the tcgen05 path (bf16 gradients, truncated basis)%s");
    if (h->dp_stage != 0) return fail(h, GLR_EINVAL, "glr_dp_begin: the previous data-parallel step is not finished%s");
    if (!G) return fail(h, GLR_EINVAL, "null gradient array%s");
    for (int i = 0; i < h->N; ++i)
        if (!G[i] || !aligned16(G[i]))
            return fail(h, GLR_EINVAL, "gradient %s is null or not 16-byte aligned", std::to_string(i).c_str());
    const int rc = dp_begin(h, G, static_cast<cudaStream_t>(stream), out);
    if (rc == GLR_OK) h->dp_stage = 1;
    return rc;
}

int glr_dp_select(glr_handle* h, void* stream, glr_dp_exchange* out) {
    if (!h || !out) return fail(h, GLR_EINVAL, "null handle or exchange descriptor%s");
    *out = glr_dp_exchange{};
    if (h->dp_stage != 1) return fail(h, GLR_EINVAL, "glr_dp_select needs a step begun by glr_dp_begin%s");
    const int rc = dp_select(h, static_cast<cudaStream_t>(stream), out);
    if (rc == GLR_OK) h->dp_stage = 2;
    return rc;
}

int glr_dp_finish(glr_handle* h, float* X, void* stream) {
    if (!h) return GLR_EINVAL;
    if (h->dp_stage != 2) return fail(h, GLR_EINVAL, "glr_dp_finish needs a step selected by glr_dp_select%s");
    if (!X || !aligned16(X)) return fail(h, GLR_EINVAL, "X is null or not 16-byte aligned%s");
    const int rc = dp_finish(h, X, static_cast<cudaStream_t>(stream));
    h->dp_stage = 0;
    return rc;
}

int glr_step_group_host(glr_handle* const* handles, int32_t count, const void* const* const* G_host,
                        float* const* X, float* const* X_host_out, void* stream) {
    if (!handles || count < 1 || !G_host || !X) return fail(nullptr, GLR_EINVAL, "null arrays or count < 1%s");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    std::vector<std::vector<const void*>> Gd(count);
    std::vector<const void* const*> Garr(count);
    std::vector<int> parity(count);
    for (int j = 0; j < count; ++j) {           // staging, streams and events on first use
        glr_handle* h = handles[j];
        if (!h) return fail(nullptr, GLR_EINVAL, "null handle in the group%s");
        if (!G_host[j] || !X[j]) return fail(h, GLR_EINVAL, "null host gradient array or X%s");
        for (int i = 0; i < h->N; ++i)
            if (!G_host[j][i]) return fail(h, GLR_EINVAL, "host gradient %s is null", std::to_string(i).c_str());
        if (!h->cstream) {
            const size_t bytes = static_cast<size_t>(h->m) * h->n * h->gsize;
            for (int b = 0; b < 2; ++b) {
                char* p = nullptr;
                const int rc = alloc(h, &p, bytes * h->N);
                if (rc != GLR_OK) return rc;
                h->Gstage2[b] = p;
            }
            if (cudaStreamCreateWithFlags(&h->cstream, cudaStreamNonBlocking) != cudaSuccess ||
                cudaEventCreateWithFlags(&h->cdone, cudaEventDisableTiming) != cudaSuccess ||
                cudaEventCreateWithFlags(&h->sfree[0], cudaEventDisableTiming) != cudaSuccess ||
                cudaEventCreateWithFlags(&h->sfree[1], cudaEventDisableTiming) != cudaSuccess ||
                cudaStreamCreateWithFlags(&h->xstream, cudaStreamNonBlocking) != cudaSuccess ||
                cudaEventCreateWithFlags(&h->xready, cudaEventDisableTiming) != cudaSuccess ||
                cudaEventCreateWithFlags(&h->xdone, cudaEventDisableTiming) != cudaSuccess)
                return fail(h, GLR_ECUDA, "could not create the host-copy streams%s");
            // alloc's zero fill runs on the legacy default stream, which the non-blocking copy
            // stream does not wait for: finish it before the first copy
            GLR_CK(h, cudaDeviceSynchronize());
        }
    }
    // every gradient copy of the call on one stream (the first handle's) and every read-back on
    // another: one stream per direction keeps the two directions on separate copy engines, so
    // the read-back of this step runs beside the next step's gradient copies
    glr_handle* h0 = handles[0];
    cudaStream_t cs = h0->cstream, xs = h0->xstream;
    for (int j = 0; j < count; ++j) {
        glr_handle* h = handles[j];
        const size_t bytes = static_cast<size_t>(h->m) * h->n * h->gsize;
        const int b = h->host_parity;
        parity[j] = b;
        // buffer b was last read by this handle's step two calls ago
        if (h->sfree_set[b]) GLR_CK(h, cudaStreamWaitEvent(cs, h->sfree[b], 0));
        Gd[j].resize(h->N);
        for (int i = 0; i < h->N; ++i) {
            char* dst = static_cast<char*>(h->Gstage2[b]) + bytes * i;
            GLR_CK(h, cudaMemcpyAsync(dst, G_host[j][i], bytes, cudaMemcpyHostToDevice, cs));
            Gd[j][i] = dst;
        }
        Garr[j] = Gd[j].data();
    }
    GLR_CK(h0, cudaEventRecord(h0->cdone, cs));
    GLR_CK(h0, cudaStreamWaitEvent(st, h0->cdone, 0));
    const int rc = glr_step_group(handles, count, Garr.data(), X, stream);
    if (rc != GLR_OK) return rc;
    bool out = false;
    for (int j = 0; j < count; ++j) {
        glr_handle* h = handles[j];
        const int b = parity[j];
        GLR_CK(h, cudaEventRecord(h->sfree[b], st));
        h->sfree_set[b] = true;
        h->host_parity = b ^ 1;
        out = out || (X_host_out && X_host_out[j]);
    }
    if (!out) return GLR_OK;
    // the read-back after the step; only the next step's update (which rewrites X) waits for it
    GLR_CK(h0, cudaEventRecord(h0->xready, st));
    GLR_CK(h0, cudaStreamWaitEvent(xs, h0->xready, 0));
    for (int j = 0; j < count; ++j) {
        glr_handle* h = handles[j];
        if (!X_host_out[j]) continue;
        GLR_CK(h, cudaMemcpyAsync(X_host_out[j], X[j], sizeof(float) * h->m * h->n, cudaMemcpyDeviceToHost, xs));
        GLR_CK(h, cudaEventRecord(h->xdone, xs));
        h->x_pending = true;
    }
    return GLR_OK;
}

}  // extern "C"
