// bsr_spmm_noalloc: the BSR product for callers that cannot allocate device
// memory (inside a CUDA graph capture, under a fixed memory budget or their
// own allocator, or where an allocation's implicit synchronisation is not
// acceptable). Split-row partial tiles go to a fixed scratch array compiled
// into this file instead of the handle's workspace; the call allocates
// nothing. See include/bsr.h for the contract.
#include <mutex>
#include <unordered_map>

#include "bsr_internal.h"
#include "schedule.h"

namespace {

// Scratch for split-row partials, one copy per device that loads the library.
__device__ __align__(256) float g_noalloc_scratch[BSR_NOALLOC_SCRATCH_BYTES / sizeof(float)];

std::mutex g_mu;
std::unordered_map<int, float *> g_scratch;   // device -> device address of g_noalloc_scratch

// Device address of the scratch array on `device` (which must be current).
// In host code the array's name is only a host-side stand-in, so the address
// is looked up once per device and kept.
bsr_status_t scratch_on(int device, float **out) {
    std::lock_guard<std::mutex> lk(g_mu);
    auto it = g_scratch.find(device);
    if (it != g_scratch.end()) {
        *out = it->second;
        return BSR_OK;
    }
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) {
        cudaGetLastError();
        return BSR_ERR_CUDA;
    }
    g_scratch[device] = static_cast<float *>(p);
    *out = static_cast<float *>(p);
    return BSR_OK;
}

bool is_device_ptr(const void *p, int device) {
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return (at.type == cudaMemoryTypeDevice && at.device == device) || at.type == cudaMemoryTypeManaged;
}

bool overlap(const void *a, size_t na, const void *b, size_t nb) {
    const uintptr_t x = (uintptr_t)a, y = (uintptr_t)b;
    return na && nb && x < y + nb && y < x + na;
}

}  // namespace

extern "C" bsr_status_t bsr_spmm_noalloc(bsr_handle_t h, const void *X, const float *bias, void *Y, int64_t N,
                                         void *stream) {
    if (!h || N < 0) return BSR_ERR_INVALID_ARG;
    if (N == 0) return BSR_OK;
    if (!X || !Y) return BSR_ERR_INVALID_ARG;
    const bsr::Schedule &sc = *h->sched;
    // the split-row partials of this call must fit the scratch array
    if ((double)sc.n_slots * (double)N * sc.ex_R * 4.0 > (double)BSR_NOALLOC_SCRATCH_BYTES) return BSR_ERR_CAPACITY;
    const size_t es = bsr::dtype_size(h->dt);
    const size_t xbytes = (size_t)N * h->K * es, ybytes = (size_t)N * h->M * es;
    if ((uintptr_t)X % 16 || (uintptr_t)Y % 16 || (uintptr_t)bias % 4) return BSR_ERR_ALIGNMENT;
    if (overlap(X, xbytes, Y, ybytes) || (bias && overlap(bias, (size_t)h->M * 4, Y, ybytes)))
        return BSR_ERR_INVALID_ARG;

    int prev = -1;
    if (cudaGetDevice(&prev) != cudaSuccess) {
        cudaGetLastError();
        return BSR_ERR_CUDA;
    }
    if (prev != h->device && cudaSetDevice(h->device) != cudaSuccess) {
        cudaGetLastError();
        return BSR_ERR_CUDA;
    }
    bsr_status_t st = BSR_OK;
    float *scratch = nullptr;
    if ((xbytes && !is_device_ptr(X, h->device)) || (ybytes && !is_device_ptr(Y, h->device)) ||
        (bias && !is_device_ptr(bias, h->device))) {
        st = BSR_ERR_INVALID_ARG;
    } else {
        st = scratch_on(h->device, &scratch);
    }
    if (st == BSR_OK) {
        bsr::LaunchArgs a{&sc,   h->data_packed ? h->data_packed : h->data,
                          X,     bias,
                          Y,     scratch,
                          h->d_status, N,
                          static_cast<cudaStream_t>(stream), h->wait_ns,
                          h->stall_chunk};
        if (bsr::launch_spmm(a) != cudaSuccess) {
            cudaGetLastError();
            st = BSR_ERR_CUDA;
        }
    }
    if (prev != h->device) cudaSetDevice(prev);
    return st;
}
