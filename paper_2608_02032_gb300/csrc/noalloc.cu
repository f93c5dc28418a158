// dart_sma_forward_noalloc: state-memory attention and the gated merge for
// callers that cannot allocate device memory and cannot hand the library a
// workspace either. Some host frameworks give a plugin only its input and
// output buffers and own every other byte of device memory. Some
// latency-critical services forbid allocation once they have started, because
// cudaMalloc and cudaFree can synchronise the device. Some processes run
// under a fixed device-memory budget.
//
// The only scratch the computation needs is the inverse RMS of every memory
// row (what dart_sma_forward computes into its workspace when rM is NULL). Here
// it lives in a file-scope device array of fixed size, so this entry point
// needs no allocation from anyone.
#include <mutex>

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "dart.h"
#include "kernels.h"

namespace {

// Scratch for r (one fp32 per memory row). Every GPU that loads the library
// holds these 4 MiB until the process exits.
constexpr long long kNoallocRows = 1LL << 20;
__device__ __align__(256) float g_noalloc_rms[kNoallocRows];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
float* g_scratch_ptr[kMaxDevices] = {};  // device address of g_noalloc_rms, per device

// Device address of the scratch on the current device. In host code
// g_noalloc_rms names a host-side stand-in, not device memory, so the address
// has to come from cudaGetSymbolAddress, once per device, with that device
// current.
cudaError_t scratch_on_current_device(float** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (g_scratch_ptr[dev] == nullptr) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_rms);
        if (e != cudaSuccess) return e;
        g_scratch_ptr[dev] = static_cast<float*>(p);
    }
    *out = g_scratch_ptr[dev];
    return cudaSuccess;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

}  // namespace

extern "C" dart_status dart_sma_forward_noalloc(const dart_dims* d, const void* M, const void* Q,
                                                const void* Cm, const void* E, const void* z,
                                                const void* Y_ssd, void* Y, void* R, float* lse,
                                                void* stream) {
    const dart_status st = dart::validate_dims(d, true);
    if (st != DART_OK) return st;
    const void* req[] = {M, Q, Cm, E, z, Y_ssd, Y};
    for (const void* p : req)
        if (p == nullptr || !aligned16(p)) return DART_ERR_INVALID_ARG;
    if ((R && !aligned16(R)) || (lse && !aligned16(lse))) return DART_ERR_INVALID_ARG;
    const long long rows = d->batch * (d->seqlen / d->chunk) * d->nheads * d->dstate;
    if (rows > kNoallocRows) return DART_ERR_TOO_LARGE;

    float* r = nullptr;
    cudaError_t e = scratch_on_current_device(&r);
    if (e != cudaSuccess) return dart::record_cuda_error(e);
    // Every entry of r that the SMA kernel reads is written first, so nothing
    // needs clearing; the array keeps whatever the last call left in it.
    cudaStream_t s = (cudaStream_t)stream;
    e = d->mem_dtype == DART_F32
            ? dart::launch_memory_rms<float>(M, r, rows, d->headdim, d->eps, s)
            : dart::launch_memory_rms<__nv_bfloat16>(M, r, rows, d->headdim, d->eps, s);
    if (e != cudaSuccess) return dart::record_cuda_error(e);
    // The rest is the FFMA SMA kernel of dart_sma_forward with the r computed
    // above (it needs no scratch beyond r).
    dart::SmaArgs a{};
    a.B = d->batch; a.L = d->seqlen; a.H = d->nheads; a.G = d->ngroups;
    a.P = d->headdim; a.N = d->dstate; a.S = d->chunk; a.eps = d->eps;
    a.M = M; a.rM = r; a.Q = Q; a.Cm = Cm; a.E = E; a.z = z; a.Yssd = Y_ssd; a.Y = Y; a.R = R;
    a.lse = lse;
    typedef __nv_bfloat16 bf;
    if (d->in_dtype == DART_F32)
        e = dart::launch_sma_forward_simt<float, float, float>(a, s);
    else if (d->mem_dtype == DART_F32)
        e = dart::launch_sma_forward_simt<bf, float, float>(a, s);
    else if (d->out_dtype == DART_F32)
        e = dart::launch_sma_forward_simt<bf, bf, float>(a, s);
    else
        e = dart::launch_sma_forward_simt<bf, bf, bf>(a, s);
    return e == cudaSuccess ? DART_OK : dart::record_cuda_error(e);
}
