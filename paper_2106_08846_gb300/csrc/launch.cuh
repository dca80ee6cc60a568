// Kernel launches of the product path.
//
// Every product kernel is launched with programmatic stream serialisation:
// the kernel lets the next kernel of its stream be scheduled as soon as all
// of its own CTAs are running (griddepcontrol.launch_dependents at entry),
// and the next kernel runs its prologue -- barrier set-up, fetching the
// handle's own schedule and block values -- on the SMs that free up, then
// waits (griddepcontrol.wait) before it touches anything an earlier kernel
// may write: X, the bias, Y and the split-row workspace. A chain of products
// on one stream (layers, or the block-shape sweep) thus overlaps each
// kernel's start with the previous one's tail, with the stream's ordering
// intact. BSR_PDL=0 in the environment turns it off (plain stream order).
#pragma once

#include <cuda_runtime.h>

#include <cstdlib>
#include <utility>

namespace bsr {

inline bool pdl_enabled() {
    static const bool on = [] {
        const char *v = std::getenv("BSR_PDL");
        return !(v && v[0] == '0');
    }();
    return on;
}

// Launch `kernel` on `s`.
template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                          Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    unsigned n = 0;
    if (pdl_enabled()) {
        attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[n].val.programmaticStreamSerializationAllowed = 1;
        n++;
    }
    cfg.attrs = attr;
    cfg.numAttrs = n;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

}  // namespace bsr
