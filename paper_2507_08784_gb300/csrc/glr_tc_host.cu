// Host side of the tcgen05 large-matrix path (k_tc.cu): which handles take it, the buffers it adds
// to a handle's state and the table of tensor maps (tile-copy descriptors) of its operands.
#include "glr_host.cuh"

namespace glr {
namespace host {

namespace {
inline int up32(int x) { return (x + 31) & ~31; }
}  // namespace

// The path needs a truncated basis, bf16 gradients (its TF32 products are checked against the
// 2e-2 bf16 tolerance), MSGD or Adam (the optimizers its update epilogue fuses), rows of 16-byte
// multiples for every tile copy (m', n' multiples of 8, r, k of 4), at most 8 nodes (N x 64 accumulator
// columns), 16 <= r <= 128 (the projected mean takes one 128-row tile), k <= 256 (one MMA's N)
// and m' >= 128 (one MMA's M).
// A truncated refresh's k x k Rayleigh-Ritz eigenproblem goes to the blocked Jacobi when k is a
// multiple of 128 from 256 (its pairs are 128 x 128); smaller k stay on the one-CTA solver.
bool tcl_rr_blocked(const glr_handle* h) { return !h->exact && h->k >= 256 && h->k % 128 == 0; }

bool tcl_eligible(int64_t mp, int64_t np, int r, int N, int k, bool exact, const glr_schedule* s) {
    if (s->grad_dtype != GLR_BF16) return false;
    // the full basis takes this path above m' = 1024 only (the blocked Jacobi's 128-index pairs)
    if (exact && (mp <= kMaxFullBasis || mp > kBjacMaxN || mp % 128)) return false;
    if (s->optimizer != GLR_MSGD && s->optimizer != GLR_ADAM) return false;
    if (mp % 8 || np % 8 || r % 4 || k % 4) return false;   // bf16 rows of 16-byte multiples too
    if (N > 8 || r < 16 || r > 128 || (!exact && k > 256)) return false;
    return mp >= 128;
}

int tcl_alloc(glr_handle* h) {
    const size_t MP = h->mp, NP = h->np;
    h->rpad = up32(h->r);
    h->kpad = up32(h->k);
    // PrevProj node groups: na nodes per tile (na x rpad accumulator columns, two stages of
    // na 16 KiB slices plus the rpad x 32 slice of P^T)
    int na_max = std::min(512 / h->rpad, static_cast<int>((110 * 1024 - (size_t)h->rpad * 128) / 16384));
    na_max = std::max(1, std::min(na_max, h->N));
    h->tc_ng = (h->N + na_max - 1) / na_max;
    h->tc_na = (h->N + h->tc_ng - 1) / h->tc_ng;
    h->tc_lam_tiles = 4 * ((h->np + 127) / 128);   // one partial per 32 columns
    int rc = GLR_OK;
    auto A = [&](float** p, size_t cnt) { if (rc == GLR_OK) rc = alloc(h, p, cnt); };
    A(&h->PT0, (size_t)h->rpad * MP);
    A(&h->PT1, (size_t)h->rpad * MP);
    if (h->exact) {
        A(&h->UT, MP * MP);
    } else {
        A(&h->WT, NP * h->kpad);
        A(&h->YTk, (size_t)h->kpad * MP);
    }
    A(&h->RbarT, NP * h->rpad);
    h->Pbuf0 = h->P;
    return rc;
}

float* tcl_PT_of(const glr_handle* h, const float* P) { return P == h->Pbuf0 ? h->PT0 : h->PT1; }
const CUtensorMap* tcl_map(const glr_handle* h, int which) { return h->dmaps + which; }
const CUtensorMap* tcl_map_P(const glr_handle* h, const float* P) { return h->dmaps + (P == h->Pbuf0 ? kMapP0 : kMapP1); }
const CUtensorMap* tcl_map_PT(const glr_handle* h, const float* P) {
    return h->dmaps + (P == h->Pbuf0 ? kMapPT0 : kMapPT1);
}

// Every map: fp32, 128-byte swizzle, boxes 32 elements wide (one 128-byte K slice); dims and
// strides innermost first, strides in bytes for dimensions 1.. .
int tcl_maps(glr_handle* h) {
    const uint64_t mp = h->mp, np = h->np, N = h->N, r = h->r, k = h->k;
    const uint64_t rp = h->rpad, kp = h->kpad;
    {   // refresh scratch, allocated after the checkpointed state
        int rc = GLR_OK;
        auto A = [&](float** p, size_t cnt) { if (rc == GLR_OK) rc = alloc(h, p, cnt); };
        if (h->exact) {
            A(&h->Vbuf2, mp * mp); A(&h->bjJ, mp * 128); A(&h->bjJlo, mp * 128);
            A(&h->Hlo, mp * mp); A(&h->Ttlo, mp * mp); A(&h->Vlo, mp * mp); A(&h->V2lo, mp * mp);
            A(&h->bjpart, (size_t)2 * kBjacNormCtas * kBjacGroupMax);
        } else {
            const size_t nch = (np + tc::kGramChunk - 1) / tc::kGramChunk;
            A(&h->Mrow, mp * np); A(&h->Mlo, mp * np);
            A(&h->QTt, kp * mp); A(&h->ZTt, kp * np);
            A(&h->gpart, std::max<size_t>(nch, 1) * kp * kp); A(&h->Linv, kp * kp);
            if (tcl_rr_blocked(h)) {        // the k x k Rayleigh-Ritz problem by the blocked Jacobi
                A(&h->Hbuf, k * k); A(&h->Hlo, k * k); A(&h->jwork, k * k); A(&h->Ttlo, k * k);
                A(&h->Vbuf, k * k); A(&h->Vlo, k * k); A(&h->Vbuf2, k * k); A(&h->V2lo, k * k);
                A(&h->bjJ, k * 128); A(&h->bjJlo, k * 128);
                A(&h->bjpart, (size_t)2 * kBjacNormCtas * kBjacGroupMax);
            }
        }
        if (rc != GLR_OK) return rc;
    }
    std::vector<CUtensorMap> maps(kNumTcMaps);
    float* Pother = h->P == h->Pbuf0 ? h->Pprev : h->P;
    bool ok = true;
    auto m2 = [&](int idx, const float* base, uint64_t d0, uint64_t d1, uint64_t ld, uint32_t box1) {
        const uint64_t dims[2] = {d0, d1}, str[1] = {ld * 4};
        const uint32_t box[2] = {32, box1};
        ok = ok && encode_f32_map(&maps[idx], base, 2, dims, str, box);
    };
    auto m3 = [&](int idx, const float* base, uint64_t d0, uint64_t d1, uint64_t d2, uint32_t box1) {
        const uint64_t dims[3] = {d0, d1, d2}, str[2] = {d0 * 4, d0 * d1 * 4};
        const uint32_t box[3] = {32, box1, 1};
        ok = ok && encode_f32_map(&maps[idx], base, 3, dims, str, box);
    };
    m3(kMapBt, h->B, mp, np, N, 128);                      // B_i^T: n' x m' per node
    m2(kMapPT0, h->PT0, mp, rp, mp, (uint32_t)rp);         // P^T of each projector allocation
    m2(kMapPT1, h->PT1, mp, rp, mp, (uint32_t)rp);
    m2(kMapP0, h->Pbuf0, r, mp, r, 128);                   // P, row-major m' x r
    m2(kMapP1, Pother, r, mp, r, 128);
    m3(kMapRwT, h->Rw, rp, np, N, (uint32_t)tc::compose_bn());   // R_w,i^T: n' x rpad per node
    m2(kMapMbarT, h->Mbar, mp, np, mp, 128);               // Mbar^T: n' x m'
    m2(kMapRbarT, h->RbarT, rp, np, rp, 128);              // Rbar^T: n' x rpad
    if (h->exact) {
        m2(kMapUT, h->UT, mp, mp, mp, 128);                // U^T (TF32), row-major m' x m'
        m3(kMapMbar3, h->Mbar, mp, np, 1, 128);            // Mbar^T as a one-node B^T
    }
    if (h->bjJ) {
        // the blocked Jacobi's operands (rows of 128, K slices of 32) and their TF32 low parts; its
        // problem is n = m' for the full basis, k for a truncated refresh's Rayleigh-Ritz step
        const uint64_t bn = h->exact ? mp : k;
        m2(kMapBjH, h->Hbuf, bn, bn, bn, 128);  m2(kMapBjHlo, h->Hlo, bn, bn, bn, 128);
        m2(kMapBjT, h->jwork, bn, bn, bn, 128); m2(kMapBjTlo, h->Ttlo, bn, bn, bn, 128);
        m2(kMapBjV0, h->Vbuf, bn, bn, bn, 128); m2(kMapBjV0lo, h->Vlo, bn, bn, bn, 128);
        m2(kMapBjV1, h->Vbuf2, bn, bn, bn, 128); m2(kMapBjV1lo, h->V2lo, bn, bn, bn, 128);
        m2(kMapBjJ, h->bjJ, 128, bn, 128, 128); m2(kMapBjJlo, h->bjJlo, 128, bn, 128, 128);
    }
    if (!h->exact) {
    m2(kMapYT, h->YTk, mp, kp, mp, (uint32_t)kp);          // Y^T: kpad x m'
    m2(kMapYt, h->Yt, k, mp, k, 128);                      // Yt, row-major m' x k
    m2(kMapWT, h->WT, kp, np, kp, 128);                    // W^T: n' x kpad
    m2(kMapY, h->Y, k, mp, k, 128);                        // Y, row-major m' x k
    m2(kMapYtJn, h->YtJ, k, r, k, (uint32_t)rp);           // Yt[J, :] (r x k) as the N operand
    m2(kMapYtJm, h->YtJ, k, r, k, 128);                    // ... and as the M operand
    // the refresh products
    m2(kMapMrow, h->Mrow, np, mp, np, 128);                // Mbar row-major: m' x n'
    m2(kMapMlo, h->Mlo, np, mp, np, 128);                  // its TF32 low parts
    m2(kMapQTtA, h->QTt, mp, kp, mp, 128);                 // Q^T (kpad x m') in 128-row slices
    m2(kMapQTtB, h->QTt, mp, kp, mp, (uint32_t)kp);        // ... and whole (the N operand)
    m2(kMapZTtA, h->ZTt, np, kp, np, 128);                 // Z^T (kpad x n')
    m2(kMapZTtB, h->ZTt, np, kp, np, (uint32_t)kp);
    h->Qbuf0 = h->Q;
    m2(kMapQA, h->Q, k, mp, k, 128);                       // Q (either allocation), Z row-major (rows x k) as A
    m2(kMapQA1, h->Qn, k, mp, k, 128);
    m2(kMapZA, h->Z, k, np, k, 128);
    m2(kMapLinv, h->Linv, kp, kp, kp, (uint32_t)kp);       // L^{-1}, row-major kpad x kpad
    }
    // epilogue data tiles (no swizzle unless noted)
    auto plain = [&](int idx, const void* base, int rank, const uint64_t* dims, const uint64_t* str, const uint32_t* box,
                     CUtensorMapSwizzle swz) {
        ok = ok && encode_map(&maps[idx], CU_TENSOR_MAP_DATA_TYPE_FLOAT32, base, rank, dims, str, box, swz);
    };
    {
        const uint64_t d3[3] = {mp, np, N}, s3[2] = {mp * 4, mp * np * 4};
        const uint32_t b3[3] = {128, 64, 1};
        plain(kMapBtD, h->B, 3, d3, s3, b3, CU_TENSOR_MAP_SWIZZLE_NONE);          // B_i^T tiles, 128 x 64
        const uint64_t d2[2] = {mp, np}, s2[1] = {mp * 4};
        const uint32_t bl[2] = {128, 128}, bu[2] = {128, 32};
        plain(kMapMbarL, h->Mbar, 2, d2, s2, bl, CU_TENSOR_MAP_SWIZZLE_NONE);     // Mbar^T tiles, 128 x 128
        plain(kMapMbarU, h->Mbar, 2, d2, s2, bu, CU_TENSOR_MAP_SWIZZLE_NONE);     // ... 128 rows x 32 columns
        for (int q = 0; q < 2; ++q) {                                            // Mo, Vo in X's layout
            const float* base = q ? h->Vo : h->Mo;
            if (!base) continue;
            if (h->transposed) {
                const uint64_t dx[2] = {mp, np}, sx[1] = {mp * 4};
                const uint32_t bx[2] = {128, 32};
                plain(q ? kMapVo : kMapMo, base, 2, dx, sx, bx, CU_TENSOR_MAP_SWIZZLE_NONE);
            } else {
                const uint64_t dx[2] = {np, mp}, sx[1] = {np * 4};
                const uint32_t bx[2] = {32, 128};
                plain(q ? kMapVo : kMapMo, base, 2, dx, sx, bx, CU_TENSOR_MAP_SWIZZLE_128B);
            }
        }
    }
    if (!ok) return fail(h, GLR_ECUDA, "could not describe the operands for tile copies%s");
    CUtensorMap* d = nullptr;
    int rc = alloc(h, &d, maps.size() + 2 * (size_t)h->N + 2);
    if (rc != GLR_OK) return rc;
    GLR_CK(h, cudaMemcpy(d, maps.data(), sizeof(CUtensorMap) * maps.size(), cudaMemcpyHostToDevice));
    h->dmaps = d;
    return GLR_OK;
}

// The maps of this step's N gradients (bf16 tiles of 128 rows x 64 columns, read in the caller's
// layout): one of two slots, re-encoded and copied to the device (stream-ordered) only when the
// set of pointers differs from both.
const CUtensorMap* tcl_grad_maps(glr_handle* h, const void* const* G, cudaStream_t st, int* rc) {
    *rc = GLR_OK;
    for (int q = 0; q < 2; ++q) {
        bool same = true;
        for (int i = 0; i < h->N && same; ++i) same = h->tc_gptr[q][i] == G[i];
        if (same) { h->tc_glast = q; return h->dmaps + kNumTcMaps + q * h->N; }
    }
    const int q = h->tc_glast ^ 1;
    std::vector<CUtensorMap> maps(h->N);
    const uint64_t mp = h->mp, np = h->np;
    for (int i = 0; i < h->N; ++i) {
        bool ok;
        if (h->transposed) {                       // G is n' x m' row-major: G(a, c) = G[c m' + a]
            const uint64_t d[2] = {mp, np}, s[1] = {mp * 2};
            const uint32_t b[2] = {128, 64};
            ok = encode_map(&maps[i], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, G[i], 2, d, s, b, CU_TENSOR_MAP_SWIZZLE_NONE);
        } else {
            const uint64_t d[2] = {np, mp}, s[1] = {np * 2};
            const uint32_t b[2] = {64, 128};
            ok = encode_map(&maps[i], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, G[i], 2, d, s, b, CU_TENSOR_MAP_SWIZZLE_128B);
        }
        if (!ok) {
            *rc = fail(h, GLR_ECUDA, "could not describe gradient %s for tile copies", std::to_string(i).c_str());
            return nullptr;
        }
    }
    CUtensorMap* dst = h->dmaps + kNumTcMaps + q * h->N;
    const cudaError_t e = cudaMemcpyAsync(dst, maps.data(), sizeof(CUtensorMap) * h->N, cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) { *rc = fail_cuda(h, e, __FILE__, __LINE__); return nullptr; }
    for (int i = 0; i < h->N; ++i) h->tc_gptr[q][i] = G[i];
    h->tc_glast = q;
    return dst;
}

// The map of X (fp32 tiles of 128 x 32 in X's layout, as Mo and Vo), cached like the gradients'.
const CUtensorMap* tcl_x_map(glr_handle* h, const float* X, cudaStream_t st, int* rc) {
    *rc = GLR_OK;
    CUtensorMap* slots = h->dmaps + kNumTcMaps + 2 * h->N;
    for (int q = 0; q < 2; ++q)
        if (h->tc_xptr[q] == X) { h->tc_xlast = q; return slots + q; }
    const int q = h->tc_xlast ^ 1;
    const uint64_t mp = h->mp, np = h->np;
    CUtensorMap map;
    bool ok;
    if (h->transposed) {
        const uint64_t d[2] = {mp, np}, s[1] = {mp * 4};
        const uint32_t b[2] = {128, 32};
        ok = encode_map(&map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, X, 2, d, s, b, CU_TENSOR_MAP_SWIZZLE_NONE);
    } else {
        const uint64_t d[2] = {np, mp}, s[1] = {np * 4};
        const uint32_t b[2] = {32, 128};
        ok = encode_map(&map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, X, 2, d, s, b, CU_TENSOR_MAP_SWIZZLE_128B);
    }
    if (!ok) { *rc = fail(h, GLR_ECUDA, "could not describe X for tile copies%s"); return nullptr; }
    const cudaError_t e = cudaMemcpyAsync(slots + q, &map, sizeof(CUtensorMap), cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess) { *rc = fail_cuda(h, e, __FILE__, __LINE__); return nullptr; }
    h->tc_xptr[q] = X;
    h->tc_xlast = q;
    return slots + q;
}

}  // namespace host
}  // namespace glr
