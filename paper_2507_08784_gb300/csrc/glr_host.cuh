// Host-side internals of libglr.so shared by its translation units: the handle (the state of one
// layer matrix), error reporting, per-phase profiling, device allocation, the product dispatch
// and the refresh orchestration.  Not part of the C ABI (include/glr.h is).
#pragma once

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include <cublas_v2.h>

#include "glr_internal.cuh"

struct glr_handle {
    int64_t m = 0, n = 0;
    int mp = 0, np = 0, transposed = 0, r = 0, N = 0, k = 0, exact = 0;
    glr_schedule s{};
    int device = 0;
    size_t gsize = 4;
    // device state
    float *B = nullptr, *Mbar = nullptr, *Rw = nullptr, *Rbar = nullptr, *P = nullptr, *Pprev = nullptr;
    int32_t* J = nullptr;
    float *lam = nullptr, *lam_part = nullptr;
    int ntiles = 0;                 // lambda tiles of the first-path kernel (64 columns)
    int fused = 0, BN = 0, nstrips = 0;   // fused strip kernels: strip width, strips per matrix
    int mma = 0;                          // compose on the tensor cores (k_mma.cu)
    int tma = 0;                          // ... with its ring filled by tile copies
    CUtensorMap Bmap{};                   // tile-copy descriptor of B (n' x m' x N)
    struct GMap { const void* ptr; CUtensorMap map; };
    std::vector<GMap> gmaps;              // per node: the descriptors of its last two gradient buffers
    float *Mo = nullptr, *Vo = nullptr;
    float *U = nullptr, *Hbuf = nullptr, *Vbuf = nullptr, *evals = nullptr, *evals_sorted = nullptr;
    float *Q = nullptr, *Qn = nullptr, *Y = nullptr, *Yt = nullptr, *T = nullptr, *dsign = nullptr;
    float *Wbar = nullptr, *Z = nullptr, *Zn = nullptr, *Hk = nullptr, *Vk = nullptr, *gram = nullptr, *scratch = nullptr;
    float *YT = nullptr, *YtT = nullptr;   // k x transposed_pitch(m') copies of Y and Yt for the fused kernel
    float *YF = nullptr, *YtF = nullptr;   // Y and Yt in fragment order for the tensor-core kernel
    int* dflags = nullptr;   // [0] Cholesky restarts, [1] Jacobi sweeps of the last refresh,
                             // [2] bounded device waits that gave up, [3] warps that found a NaN /
                             // Inf in Mbar, [4..5] the cooperative Jacobi's grid barrier, [6]
                             // refresh factorisations that failed (GLR_ENUMERIC), [7] unused
    float* gemm_ws = nullptr;   // split-K partial tiles of the refresh GEMMs
    // Large plain products (>= 2^26 flops) go to cuBLAS: one library handle for the step stream
    // and one for the refresh stream (a handle's workspace must not serve two streams at once).
    cublasHandle_t cb[2] = {nullptr, nullptr};
    // The first path with its rank-r / rank-k products as library GEMMs (set when those products
    // are large): E_i = B_i - P_prev (P_prev^T B_i) in place, D = Mbar - Yt W and Ghat = P Rbar
    // in mn_scratch (m' x n').
    int tc = 0;
    float* mn_scratch = nullptr;
    float* jwork = nullptr;      // full basis: the grouped Jacobi's second m' x m' buffer
    float* jpart = nullptr;      // full basis: its per-CTA norm partials (used by a group's first handle)
    float* YtJ = nullptr;        // Yt[J, :] (r x k) for P = U[:, J] as a library product
    float* amsv = nullptr;       // AMSGrad: the scalar normaliser and this step's maximum of V
    float* galr = nullptr;       // Algorithm 5: the subspace step direction M / (sqrt(V) + eps), r x n'
    // The tcgen05 large-matrix path (k_tc.cu; truncated basis, bf16 gradients, MSGD / Adam): B
    // and Mbar are column-major there, P keeps a transposed copy per projector allocation, and
    // the tensor maps of every operand sit in a device table (not part of the checkpointed state).
    int tcl = 0, rpad = 0, kpad = 0, tc_na = 0, tc_ng = 0, tc_lam_tiles = 0;
    // refresh scratch of the tcgen05 path (not checkpointed): Mbar row-major and its TF32 low parts,
    // TF32 transposes of Q and Z, Gram partials, L^{-1}
    float *Mrow = nullptr, *Mlo = nullptr, *QTt = nullptr, *ZTt = nullptr, *gpart = nullptr, *Linv = nullptr;
    float* Qbuf0 = nullptr;                       // Q's first allocation (Q and Qn trade places)
    // the full basis on the tcgen05 path (m' > 1024): U^T rounded to TF32 (the score operand, part
    // of the state), and the blocked Jacobi's scratch (not checkpointed): the second V buffer, the
    // pair rotations (m' x 128), the pair solver's eigenvalues, the norm partials, the sweep count
    float *UT = nullptr, *Vbuf2 = nullptr, *bjJ = nullptr, *bjpart = nullptr;
    // ... and the TF32 low parts of the rotations' operands: J^T, H, T^T (in jwork) and both V buffers
    float *bjJlo = nullptr, *Hlo = nullptr, *Ttlo = nullptr, *Vlo = nullptr, *V2lo = nullptr;
    int bj_sweeps = 0, numeric_failures_host = 0;
    const float* bj_V = nullptr;       // the blocked Jacobi's final V (after a refresh that used it)
    // a data-parallel step in progress (glr_dp_begin / glr_dp_select / glr_dp_finish): 0 idle,
    // 1 begun, 2 selected; the step's plan and the caller's gradient pointers
    int dp_stage = 0, dp_flags = 0;
    const void* dp_G[GLR_MAX_NODES] = {};
    float* Pbuf0 = nullptr;                    // the first projector allocation (P and Pprev trade places)
    float *PT0 = nullptr, *PT1 = nullptr;      // P^T of Pbuf0 / of the other allocation (rpad x m')
    float *WT = nullptr, *YTk = nullptr, *RbarT = nullptr;   // W^T (n' x kpad), Y^T (kpad x m'), Rbar^T (n' x rpad)
    CUtensorMap* dmaps = nullptr;
    const void* tc_gptr[2][GLR_MAX_NODES] = {};   // gradient pointers described in each map slot
    const float* tc_xptr[2] = {nullptr, nullptr};
    int tc_glast = 0, tc_xlast = 0;               // the slot used last
    cudaStream_t rstream = nullptr;            // side stream of this handle's refresh
    cudaEvent_t rfork = nullptr, rdone = nullptr, rpow = nullptr;
    int pow_ok = 0;                            // refresh through the grouped power iteration (k_power.cu)
    float *powpart = nullptr, *powG = nullptr, *powS = nullptr;
    void* Gstage = nullptr;
    // glr_step_group_host: two device staging buffers of N gradients, filled on a copy stream
    void* Gstage2[2] = {nullptr, nullptr};
    cudaStream_t cstream = nullptr;
    cudaEvent_t cdone = nullptr, sfree[2] = {nullptr, nullptr};
    bool sfree_set[2] = {false, false};
    int host_parity = 0;
    // the read-back of X to the host (glr_step_group_host) on its own stream: xready marks X final
    // on the step's stream, xdone the copy's end; x_pending makes the next step's update wait
    cudaStream_t xstream = nullptr;
    cudaEvent_t xready = nullptr, xdone = nullptr;
    bool x_pending = false;
    // host state
    int64_t t = 0, refreshes = 0, comm = 0, state_bytes = 0, period_start = 0;
    bool e_zero = true, force_refresh = false, last_uncompressed = true, basis_from_user = false;
    bool has_forceJ = false, forced_this_step = false;
    std::vector<int32_t> forceJ, iotaJ;
    std::vector<void*> allocs;
    std::vector<size_t> alloc_bytes;
    size_t n_state_allocs = 0;       // allocations made by glr_create (the checkpointed state)
    std::string err;
    // launch counting and optional per-phase event timing
    int64_t launches = 0;
    bool prof = false;
    struct Rec { int phase; cudaEvent_t a, b; int64_t launches; };
    std::vector<Rec> recs;
    std::vector<cudaEvent_t> free_events;
    double prof_ms[GLR_PHASES] = {};
    int64_t prof_launch[GLR_PHASES] = {}, prof_count[GLR_PHASES] = {};
    int cur_phase = -1;
    cudaEvent_t cur_start = nullptr;
    int64_t cur_launch0 = 0;
};

namespace glr {
namespace host {

constexpr int kMaxRank = 512;
constexpr int kMaxFullBasis = 1024;
constexpr int kMaxTruncBasis = 512;

extern thread_local std::string g_create_err;   // message of the last failed glr_create
extern thread_local float* g_ws;                // split-K workspace of the handle being stepped

// Record a failure message on h (or as the last glr_create failure when h is null) and return
// code; fmt takes the string a and the integer line.
int fail(glr_handle* h, int code, const char* fmt, const char* a = "", int line = 0);
// A failed CUDA call at file:line of this library.
int fail_cuda(glr_handle* h, cudaError_t e, const char* file, int line);

#define GLR_CK(h, expr)                                                                        \
    do {                                                                                       \
        cudaError_t e__ = (expr);                                                              \
        if (e__ != cudaSuccess) return ::glr::host::fail_cuda((h), e__, __FILE__, __LINE__);     \
    } while (0)

// Count kernels launched by a launcher call and check its status.
#define GLR_LAUNCH(h, nk, expr)                                                                \
    do {                                                                                       \
        (h)->launches += (nk);                                                                 \
        GLR_CK(h, expr);                                                                       \
    } while (0)

cudaEvent_t take_event(glr_handle* h);
void phase_begin(glr_handle* h, int phase, cudaStream_t st);
void phase_end(glr_handle* h, cudaStream_t st);

struct PhaseScope {
    glr_handle* h; cudaStream_t st;
    PhaseScope(glr_handle* h_, int phase, cudaStream_t st_) : h(h_), st(st_) { phase_begin(h, phase, st); }
    ~PhaseScope() { phase_end(h, st); }
};

// Zero-filled device allocation owned by h (freed by free_all).
template <typename T>
int alloc(glr_handle* h, T** p, size_t count) {
    if (count == 0) count = 1;
    void* ptr = nullptr;
    const size_t bytes = count * sizeof(T);
    if (cudaMalloc(&ptr, bytes) != cudaSuccess) {
        cudaGetLastError();
        return fail(h, GLR_ENOMEM, "device allocation of %s bytes failed", std::to_string(bytes).c_str());
    }
    h->allocs.push_back(ptr);
    h->alloc_bytes.push_back(bytes);
    h->state_bytes += static_cast<int64_t>(bytes);
    if (cudaMemset(ptr, 0, bytes) != cudaSuccess) return fail(h, GLR_ECUDA, "cudaMemset failed%s");
    *p = static_cast<T*>(ptr);
    return GLR_OK;
}
void free_all(glr_handle* h);

// Tile-copy descriptors (the tensor-core compose's ring).
bool encode_strip_map(CUtensorMap* map, const void* base, int rows, int cols, int depth, int gsize);
bool gradient_map(glr_handle* h, int i, const void* ptr, CUtensorMap* out);

// Plain products C = alpha A B + beta C (GemmDesc semantics): gd builds the descriptor (with the
// split-K workspace g_ws), gemm runs it on cuBLAS when large, else on gemm_f32.
GemmDesc gd(int M, int N, int K, const float* A, int64_t sAi, int64_t sAp, const float* B, int64_t sBp,
            int64_t sBj, float* C, int64_t sCi, int64_t sCj, float alpha = 1.f, float beta = 0.f);
int gemm_cublas(glr_handle* h, const GemmDesc& d0, cudaStream_t st);
int gemm(glr_handle* h, const GemmDesc& d, cudaStream_t st);

#define GLR_GEMM(h, d, st)                                                                     \
    do {                                                                                       \
        const int gemm_rc_ = ::glr::host::gemm((h), (d), (st));                                \
        if (gemm_rc_ != GLR_OK) return gemm_rc_;                                               \
    } while (0)

// The tcgen05 large-matrix path (glr_tc_host.cu): eligibility, buffers, tensor maps.
enum TcMap { kMapBt, kMapPT0, kMapPT1, kMapP0, kMapP1, kMapRwT, kMapMbarT, kMapYT, kMapYt, kMapWT, kMapY, kMapYtJn,
             kMapYtJm, kMapRbarT, kMapBtD, kMapMbarL, kMapMbarU, kMapMo, kMapVo,
             kMapMrow, kMapMlo, kMapQTtA, kMapQTtB, kMapZTtA, kMapZTtB, kMapQA, kMapQA1, kMapZA, kMapLinv,
             kMapUT, kMapMbar3, kMapBjH, kMapBjHlo, kMapBjT, kMapBjTlo, kMapBjV0, kMapBjV0lo, kMapBjV1, kMapBjV1lo,
             kMapBjJ, kMapBjJlo, kNumTcMaps };
// After the fixed maps: two slots of N gradient maps, then two slots for X (the caller's buffers,
// re-described only when a pointer changes).
const CUtensorMap* tcl_grad_maps(glr_handle* h, const void* const* G, cudaStream_t st, int* rc);
const CUtensorMap* tcl_x_map(glr_handle* h, const float* X, cudaStream_t st, int* rc);
bool tcl_eligible(int64_t mp, int64_t np, int r, int N, int k, bool exact, const glr_schedule* s);
bool tcl_rr_blocked(const glr_handle* h);
int tcl_alloc(glr_handle* h);         // state buffers (before n_state_allocs is fixed)
int tcl_maps(glr_handle* h);          // the device map table (after)
float* tcl_PT_of(const glr_handle* h, const float* P);
const CUtensorMap* tcl_map(const glr_handle* h, int which);
const CUtensorMap* tcl_map_P(const glr_handle* h, const float* P);      // row-major P of that allocation
const CUtensorMap* tcl_map_PT(const glr_handle* h, const float* P);     // its transpose
bool encode_f32_map(CUtensorMap* map, const float* base, int rank, const uint64_t* dims, const uint64_t* strides,
                    const uint32_t* box);
// Any tiled map: dtype, rank (<= 3), dims innermost first, byte strides of dims 1.., box, swizzle.
bool encode_map(CUtensorMap* map, CUtensorMapDataType dtype, const void* base, int rank, const uint64_t* dims,
                const uint64_t* strides, const uint32_t* box, CUtensorMapSwizzle swz);

// The Semi-Lazy SVD refresh (glr_refresh_host.cu).
int cholqr(glr_handle* h, float*& A, float*& tmp, int rows, cudaStream_t st);
int wy_from_Q(glr_handle* h, cudaStream_t st);
int refresh_tail(glr_handle* h, cudaStream_t st);
int refresh_finish(glr_handle* h, cudaStream_t st);
int refresh_power(glr_handle* h, cudaStream_t st);
int refresh_trunc_grouped(std::vector<glr_handle*>& hs);
int refresh_tcl_grouped(std::vector<glr_handle*>& hs);    // tcgen05 path (k <= 256)
int cholqr(glr_handle* h, float*& A, float*& tmp, int rows, cudaStream_t st);
int refresh_finish(glr_handle* h, cudaStream_t st);
int refresh_grouped(std::vector<glr_handle*>& hs);
int refresh_exact_grouped(std::vector<glr_handle*>& hs);
int refresh_exact_blocked(std::vector<glr_handle*>& hs);   // m' > 1024, sorted by m'

}  // namespace host
}  // namespace glr
