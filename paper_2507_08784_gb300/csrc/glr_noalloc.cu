// glr_select_noalloc: the Approx-Top-r selection without any device allocation.
//
// Some callers cannot let a library allocate device memory: frameworks that own the whole
// GPU through their own caching allocator and forbid raw cudaMalloc from third-party code,
// services that reserve all device memory at start-up and allow no allocation on the hot
// path, and code that must not risk the device-wide synchronisation cudaMalloc/cudaFree
// can cause.  For them this entry point runs the same two kernels as glr_step's selection
// (the lambda partial sums with v_j generated in the epilogue, then the fixed-order
// reduction and arg-top-r) with its partial-sum scratch in a file-scope device array of
// fixed size instead of a handle-owned buffer.
#include <cstdio>
#include <mutex>

#include "glr_internal.cuh"

namespace {

// 2^20 floats = 4 MiB, held by every GPU that loads libglr.so until the process exits.
constexpr size_t kScratchFloats = size_t(1) << 20;
__device__ __align__(256) float g_select_scratch[kScratchFloats];

constexpr int kMaxDevices = 256;
std::mutex g_mutex;
float* g_scratch_addr[kMaxDevices] = {};   // device address of g_select_scratch, per device

}  // namespace

extern "C" int glr_select_noalloc(int32_t mp, int32_t np, int32_t r, const float* U, const float* Mbar,
                                  uint64_t seed, int64_t t, float* lambda_out, int32_t* J_out,
                                  void* stream) {
    char msg[256];
    if (mp < 1 || np < 1 || r < 1 || r > mp || mp > 16384 || !U || !Mbar || !lambda_out || !J_out) {
        glr::set_global_error("glr_select_noalloc: need 1 <= r <= m' <= 16384, n' >= 1 and non-null pointers");
        return GLR_EINVAL;
    }
    const int ntiles = (np + glr::kLambdaTile - 1) / glr::kLambdaTile;
    const size_t need = static_cast<size_t>(mp) * ntiles;
    if (need > kScratchFloats) {
        snprintf(msg, sizeof(msg),
                 "glr_select_noalloc: m' * ceil(n'/64) = %zu partial sums exceed the fixed scratch of %zu floats",
                 need, kScratchFloats);
        glr::set_global_error(msg);
        return GLR_EINVAL;
    }
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
        glr::set_global_error("glr_select_noalloc: no current CUDA device");
        return GLR_ECUDA;
    }
    float* part = nullptr;
    {
        // Host code cannot take the address of a __device__ array directly: the symbol's
        // name is a host-side stand-in.  Look the device address up once per device, with
        // that device current, and reuse it.
        std::lock_guard<std::mutex> lock(g_mutex);
        if (!g_scratch_addr[dev]) {
            void* p = nullptr;
            const cudaError_t e = cudaGetSymbolAddress(&p, g_select_scratch);
            if (e != cudaSuccess) {
                snprintf(msg, sizeof(msg), "glr_select_noalloc: cudaGetSymbolAddress failed: %s",
                         cudaGetErrorString(e));
                glr::set_global_error(msg);
                return GLR_ECUDA;
            }
            g_scratch_addr[dev] = static_cast<float*>(p);
        }
        part = g_scratch_addr[dev];
    }
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    glr::LambdaArgs la{};
    la.mode = 0; la.mp = mp; la.np = np; la.K = mp; la.A = U; la.Bm = Mbar; la.Mbar = Mbar;
    la.seed = seed; la.t = static_cast<uint32_t>(t); la.part = part; la.ntiles = ntiles;
    cudaError_t e = glr::lambda_partials(la, st);
    if (e == cudaSuccess) e = glr::select_top_r(part, ntiles, mp, r, nullptr, mp, lambda_out, J_out, st);
    if (e != cudaSuccess) {
        snprintf(msg, sizeof(msg), "glr_select_noalloc: launch failed: %s", cudaGetErrorString(e));
        glr::set_global_error(msg);
        return GLR_ECUDA;
    }
    return GLR_OK;
}
