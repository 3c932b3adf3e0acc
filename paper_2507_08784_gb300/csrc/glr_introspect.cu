// C ABI of libglr.so: checkpoints (glr_state_size / glr_save / glr_load), the forced refresh and
// selection, and the introspection calls used by tests and tools (stats, error buffers, basis,
// per-phase profiling).
#include "glr_host.cuh"

using namespace glr;
using namespace glr::host;

extern "C" {

// ---- checkpoints ---------------------------------------------------------------------------
// Layout: a header (magic, version, the handle's shape and schedule identity), the host scalars
// of the schedule, the allocation index that each role which steps swap between two buffers
// (P / Pprev, Q / Qn, Z / Zn) currently holds, then every device buffer glr_create allocated,
// in allocation order.
namespace {
constexpr uint64_t kCkptMagic = 0x31544b50524c47ull;   // "GLRPKT1"
struct CkptHeader {
    uint64_t magic, version;
    int64_t m, n;
    int32_t r, N, k, grad_dtype, optimizer, refresh_mode;
    uint64_t seed, nbuf, buf_bytes;
    int64_t t, refreshes, comm, period_start;
    int32_t e_zero, force_refresh, last_uncompressed, basis_from_user, has_forceJ, pad;
    int32_t role[6];
};
float** role_ptr(glr_handle* h, int i) {
    float** roles[6] = {&h->P, &h->Pprev, &h->Q, &h->Qn, &h->Z, &h->Zn};
    return roles[i];
}
// bytes of a checkpoint of h; a pending forced selection (r indices) is stored when has_forceJ
size_t ckpt_bytes(const glr_handle* h, bool has_forceJ) {
    size_t b = sizeof(CkptHeader) + (has_forceJ ? sizeof(int32_t) * h->r : 0);
    for (size_t i = 0; i < h->n_state_allocs; ++i) b += h->alloc_bytes[i];
    return b;
}
}  // namespace

int glr_state_size(const glr_handle* h, int64_t* bytes) {
    if (!h || !bytes) return GLR_EINVAL;
    *bytes = static_cast<int64_t>(ckpt_bytes(h, h->has_forceJ));
    return GLR_OK;
}

int glr_save(glr_handle* h, void* host_buf, int64_t bytes, void* stream) {
    if (!h) return GLR_EINVAL;
    if (!host_buf || bytes < static_cast<int64_t>(ckpt_bytes(h, h->has_forceJ)))
        return fail(h, GLR_EINVAL, "checkpoint buffer is null or smaller than glr_state_size%s");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    CkptHeader hd{};
    hd.magic = kCkptMagic; hd.version = 1;
    hd.m = h->m; hd.n = h->n; hd.r = h->r; hd.N = h->N; hd.k = h->k;
    hd.grad_dtype = h->s.grad_dtype; hd.optimizer = h->s.optimizer; hd.refresh_mode = h->s.refresh_mode;
    hd.seed = h->s.seed; hd.nbuf = h->n_state_allocs; hd.buf_bytes = ckpt_bytes(h, h->has_forceJ);
    hd.t = h->t; hd.refreshes = h->refreshes; hd.comm = h->comm; hd.period_start = h->period_start;
    hd.e_zero = h->e_zero; hd.force_refresh = h->force_refresh; hd.last_uncompressed = h->last_uncompressed;
    hd.basis_from_user = h->basis_from_user; hd.has_forceJ = h->has_forceJ;
    for (int i = 0; i < 6; ++i) {
        hd.role[i] = -1;
        float* p = *role_ptr(h, i);
        for (size_t a = 0; a < h->n_state_allocs; ++a)
            if (h->allocs[a] == p) hd.role[i] = static_cast<int32_t>(a);
    }
    char* out = static_cast<char*>(host_buf);
    std::memcpy(out, &hd, sizeof(hd));
    out += sizeof(hd);
    if (h->has_forceJ) {
        std::memcpy(out, h->forceJ.data(), sizeof(int32_t) * h->r);
        out += sizeof(int32_t) * h->r;
    }
    for (size_t a = 0; a < h->n_state_allocs; ++a) {
        GLR_CK(h, cudaMemcpyAsync(out, h->allocs[a], h->alloc_bytes[a], cudaMemcpyDeviceToHost, st));
        out += h->alloc_bytes[a];
    }
    GLR_CK(h, cudaStreamSynchronize(st));
    return GLR_OK;
}

int glr_load(glr_handle* h, const void* host_buf, int64_t bytes, void* stream) {
    if (!h) return GLR_EINVAL;
    if (!host_buf || bytes < static_cast<int64_t>(sizeof(CkptHeader)))
        return fail(h, GLR_EINVAL, "checkpoint buffer is null or too small%s");
    CkptHeader hd;
    std::memcpy(&hd, host_buf, sizeof(hd));
    if (hd.magic != kCkptMagic || hd.version != 1) return fail(h, GLR_EINVAL, "not a checkpoint of this library%s");
    if (hd.m != h->m || hd.n != h->n || hd.r != h->r || hd.N != h->N || hd.k != h->k ||
        hd.grad_dtype != h->s.grad_dtype || hd.optimizer != h->s.optimizer || hd.refresh_mode != h->s.refresh_mode ||
        hd.nbuf != h->n_state_allocs || hd.buf_bytes != ckpt_bytes(h, hd.has_forceJ != 0))
        return fail(h, GLR_EINVAL, "checkpoint of a handle with another shape or schedule%s");
    if (bytes < static_cast<int64_t>(hd.buf_bytes)) return fail(h, GLR_EINVAL, "checkpoint buffer is truncated%s");
    if (hd.seed != h->s.seed) return fail(h, GLR_EINVAL, "checkpoint of a handle with another seed%s");
    // each pair of swapped roles (P / Pprev, Q / Qn, Z / Zn) must name the two allocations this
    // handle uses for that pair, in either order
    for (int i = 0; i < 6; i += 2) {
        int cur[2] = {-1, -1};
        for (int q = 0; q < 2; ++q)
            for (size_t a = 0; a < h->n_state_allocs; ++a)
                if (h->allocs[a] == *role_ptr(h, i + q)) cur[q] = static_cast<int>(a);
        const bool same = hd.role[i] == cur[0] && hd.role[i + 1] == cur[1];
        const bool swapped = hd.role[i] == cur[1] && hd.role[i + 1] == cur[0];
        if (!same && !swapped) return fail(h, GLR_EINVAL, "checkpoint roles do not match this handle's buffers%s");
    }
    if (hd.has_forceJ != 0 && hd.has_forceJ != 1) return fail(h, GLR_EINVAL, "corrupt checkpoint header%s");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const char* in = static_cast<const char*>(host_buf) + sizeof(hd);
    if (hd.has_forceJ) {
        std::vector<int32_t> J(reinterpret_cast<const int32_t*>(in), reinterpret_cast<const int32_t*>(in) + h->r);
        for (int q = 0; q < h->r; ++q)
            if (J[q] < 0 || J[q] >= h->mp || (q && J[q] <= J[q - 1]))
                return fail(h, GLR_EINVAL, "checkpoint's pending selection is not r ascending indices in [0, m')%s");
        h->forceJ = J;
        in += sizeof(int32_t) * h->r;
    }
    for (size_t a = 0; a < h->n_state_allocs; ++a) {
        GLR_CK(h, cudaMemcpyAsync(h->allocs[a], in, h->alloc_bytes[a], cudaMemcpyHostToDevice, st));
        in += h->alloc_bytes[a];
    }
    for (int i = 0; i < 6; ++i)
        if (hd.role[i] >= 0) *role_ptr(h, i) = static_cast<float*>(h->allocs[hd.role[i]]);
    h->t = hd.t; h->refreshes = hd.refreshes; h->comm = hd.comm; h->period_start = hd.period_start;
    h->e_zero = hd.e_zero; h->force_refresh = hd.force_refresh; h->last_uncompressed = hd.last_uncompressed;
    h->basis_from_user = hd.basis_from_user; h->has_forceJ = hd.has_forceJ;
    GLR_CK(h, cudaStreamSynchronize(st));
    return GLR_OK;
}

int glr_refresh(glr_handle* h) {
    if (!h) return GLR_EINVAL;
    h->force_refresh = true;
    return GLR_OK;
}

int glr_get_stats(const glr_handle* h, glr_stats* out) {
    if (!h || !out) return GLR_EINVAL;
    out->t = h->t; out->refreshes = h->refreshes; out->comm_floats_total = h->comm;
    out->state_bytes = h->state_bytes;
    out->m_prime = h->mp; out->n_prime = h->np; out->r = h->r; out->k = h->k;
    out->transposed = h->transposed;
    int flags[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    cudaMemcpy(flags, h->dflags, sizeof(flags), cudaMemcpyDeviceToHost);
    out->last_refresh_sweeps = flags[1];
    out->launches = h->launches;
    out->path = h->tcl ? GLR_PATH_TCGEN05 : h->mma ? GLR_PATH_MMA : h->fused ? GLR_PATH_STRIP
              : h->tc ? GLR_PATH_LIBRARY : GLR_PATH_PLAIN;
    out->nonfinite = flags[3];
    out->numeric_failures = flags[6];
    return flags[2] ? GLR_ETIMEOUT : flags[6] ? GLR_ENUMERIC : flags[3] ? GLR_ENONFINITE : GLR_OK;
}

const char* glr_last_error(const glr_handle* h) { return h ? h->err.c_str() : g_create_err.c_str(); }

int glr_get_error(glr_handle* h, int32_t i, float* E_out, void* stream) {
    if (!h) return GLR_EINVAL;
    if (i < 0 || i >= h->N || !E_out) return fail(h, GLR_EINVAL, "bad node index or null output%s");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int mp = h->mp, np = h->np, r = h->r;
    float* Bi = h->B + (size_t)i * mp * np;
    float* Rwi = h->Rw + (size_t)i * r * np;
    if (h->tcl) {                              // B_i column-major: R_w,i = P_prev^T B_i with strides
        if (!h->e_zero) GLR_GEMM(h, gd(r, np, mp, h->Pprev, 1, r, Bi, 1, mp, Rwi, np, 1), st);
        GLR_LAUNCH(h, 1, tc::error_colmajor(Bi, h->Pprev, Rwi, mp, np, r, h->e_zero ? 1 : 0, E_out, st));
        return GLR_OK;
    }
    if (!h->e_zero) GLR_GEMM(h, gd(r, np, mp, h->Pprev, 1, r, Bi, np, 1, Rwi, np, 1), st);
    GLR_LAUNCH(h, 1, materialize_error(mp, np, r, h->e_zero ? 1 : 0, Bi, h->Pprev, Rwi, E_out, st));
    return GLR_OK;
}

int glr_get_selection(glr_handle* h, int32_t* J_host, float* P_out, float* Rbar_out, float* lambda_out,
                      float* Mbar_out, void* stream) {
    if (!h) return GLR_EINVAL;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const size_t mp = h->mp, np = h->np, r = h->r;
    if (P_out) GLR_CK(h, cudaMemcpyAsync(P_out, h->Pprev, 4 * mp * r, cudaMemcpyDeviceToDevice, st));
    if (Rbar_out && h->tcl)   // the tcgen05 path keeps only Rbar^T (n' x rpad)
        GLR_LAUNCH(h, 1, tc::transpose_round(Rbar_out, (int)np, h->RbarT, (int)np, (int)r, h->rpad, st));
    else if (Rbar_out) GLR_CK(h, cudaMemcpyAsync(Rbar_out, h->Rbar, 4 * r * np, cudaMemcpyDeviceToDevice, st));
    if (lambda_out) GLR_CK(h, cudaMemcpyAsync(lambda_out, h->lam, 4 * mp, cudaMemcpyDeviceToDevice, st));
    if (Mbar_out && h->tcl) GLR_LAUNCH(h, 1, transpose_pad(Mbar_out, (int)np, h->Mbar, (int)np, (int)mp, st));
    else if (Mbar_out) GLR_CK(h, cudaMemcpyAsync(Mbar_out, h->Mbar, 4 * mp * np, cudaMemcpyDeviceToDevice, st));
    if (J_host) {
        if (h->last_uncompressed) {
            for (size_t q = 0; q < r; ++q) J_host[q] = -1;
        } else {
            GLR_CK(h, cudaMemcpyAsync(J_host, h->J, 4 * r, cudaMemcpyDeviceToHost, st));
        }
    }
    GLR_CK(h, cudaStreamSynchronize(st));
    return GLR_OK;
}

int glr_get_basis(glr_handle* h, float* U_out, void* stream) {
    if (!h || !U_out) return GLR_EINVAL;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const size_t mp = h->mp;
    if (h->exact) GLR_CK(h, cudaMemcpyAsync(U_out, h->U, 4 * mp * mp, cudaMemcpyDeviceToDevice, st));
    else GLR_LAUNCH(h, 1, materialize_wy_basis(h->mp, h->k, h->Y, h->Yt, h->dsign, U_out, st));
    return GLR_OK;
}

int glr_set_basis(glr_handle* h, const float* Q, void* stream) {
    if (!h || !Q) return GLR_EINVAL;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const size_t mp = h->mp, k = h->k;
    if (h->exact) {
        GLR_CK(h, cudaMemcpyAsync(h->U, Q, 4 * mp * mp, cudaMemcpyDeviceToDevice, st));
        if (h->UT) GLR_LAUNCH(h, 1, tc::transpose_round(h->UT, (int)mp, h->U, (int)mp, (int)mp, (int)mp, st));
    } else {
        GLR_CK(h, cudaMemcpyAsync(h->Q, Q, 4 * mp * k, cudaMemcpyDeviceToDevice, st));
        int rc = wy_from_Q(h, st);
        if (rc != GLR_OK) return rc;
    }
    h->basis_from_user = true;
    return GLR_OK;
}

int glr_profile_enable(glr_handle* h, int32_t enable) {
    if (!h) return GLR_EINVAL;
    h->prof = enable != 0;
    return GLR_OK;
}

int glr_profile_read(glr_handle* h, glr_profile* out, int32_t reset) {
    if (!h || !out) return GLR_EINVAL;
    for (auto& rec : h->recs) {
        GLR_CK(h, cudaEventSynchronize(rec.b));
        float ms = 0.f;
        GLR_CK(h, cudaEventElapsedTime(&ms, rec.a, rec.b));
        h->prof_ms[rec.phase] += ms;
        h->prof_launch[rec.phase] += rec.launches;
        h->prof_count[rec.phase] += 1;
        h->free_events.push_back(rec.a);
        h->free_events.push_back(rec.b);
    }
    h->recs.clear();
    for (int p = 0; p < GLR_PHASES; ++p) {
        out->ms[p] = h->prof_ms[p];
        out->launches[p] = h->prof_launch[p];
        out->count[p] = h->prof_count[p];
        if (reset) { h->prof_ms[p] = 0.0; h->prof_launch[p] = 0; h->prof_count[p] = 0; }
    }
    return GLR_OK;
}

int glr_test_expire_wait(glr_handle* h, int32_t polls, void* stream) {
    if (!h) return GLR_EINVAL;
    if (polls < 1 || polls > (1 << 24)) return fail(h, GLR_EINVAL, "need 1 <= polls <= 2^24%s");
    GLR_LAUNCH(h, 1, tc::expire_wait(h->dflags + 2, polls, static_cast<cudaStream_t>(stream)));
    return GLR_OK;
}

int glr_force_selection(glr_handle* h, const int32_t* J_host) {
    if (!h || !J_host) return GLR_EINVAL;
    std::vector<int32_t> J(J_host, J_host + h->r);
    std::sort(J.begin(), J.end());
    for (int q = 0; q < h->r; ++q) {
        if (J[q] < 0 || J[q] >= h->mp || (q && J[q] == J[q - 1]))
            return fail(h, GLR_EINVAL, "forced selection must hold r distinct indices in [0, m')%s");
    }
    h->forceJ = J;
    h->has_forceJ = true;
    return GLR_OK;
}

}  // extern "C"
