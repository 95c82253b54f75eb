// hatq_layer_noalloc: hatq_layer for callers that cannot allocate device
// memory (for example code running where cudaMalloc is forbidden or
// unavailable: inside a host callback, a plugin whose host engine owns all
// allocations, or a caller with no memory allocator of its own). The INT8
// operand that hatq_layer stages in caller-provided scratch is staged here in
// a fixed file-scope device array instead.
//
// The array is HATQ_NOALLOC_MAX_BYTES bytes on every device that loads this
// library and stays allocated until the process exits. All calls share it and
// it keeps the last call's contents (every byte a call uses is overwritten
// before it is read, so nothing needs clearing); calls whose work overlaps on
// the GPU (different streams without ordering between them) race on it.
#include <cuda_runtime.h>

#include <atomic>

#include "hatq.h"
#include "hatq_internal.h"

namespace {

static __device__ __align__(256) int8_t g_noalloc_operand[HATQ_NOALLOC_MAX_BYTES];

// Device address of g_noalloc_operand per device, looked up once with that
// device current (in host code the symbol itself is only a host-side stand-in).
// Host threads may call concurrently: each slot is an atomic, and two threads
// that race on the first lookup store the same address. The cached address
// belongs to the device's primary context: after cudaDeviceReset() it is
// stale, as is every other device pointer the caller held.
std::atomic<int8_t *> g_operand_ptr[64];

hatq_status operand_buffer(int8_t **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return HATQ_ERR_CUDA;
    int8_t *p = g_operand_ptr[dev].load(std::memory_order_acquire);
    if (!p) {
        void *q = nullptr;
        if (cudaGetSymbolAddress(&q, g_noalloc_operand) != cudaSuccess || q == nullptr) return HATQ_ERR_CUDA;
        p = static_cast<int8_t *>(q);
        g_operand_ptr[dev].store(p, std::memory_order_release);
    }
    *out = p;
    return HATQ_OK;
}

}  // namespace

extern "C" hatq_status hatq_layer_noalloc(const void *x, int x_kind, float s_in, int n, int h, int w,
                                          const hatq_prepared *L, void *y, hatq_stream stream) {
    if (!L || n < 0 || h < 0 || w < 0 || hatq_layer_launches(x_kind, s_in, L) <= 1)
        // nothing to stage (x is already the operand) or invalid: hatq_layer decides
        return hatq_layer(x, x_kind, s_in, n, h, w, L, y, nullptr, 0, stream);
    const unsigned long long need = (unsigned long long)n * h * w * (unsigned long long)L->d.c_in;
    if (need > HATQ_NOALLOC_MAX_BYTES)
        return hatq::report(HATQ_ERR_INVALID_ARG, "hatq_layer_noalloc: the layer operand needs more bytes than the "
                                                  "fixed staging array holds (HATQ_NOALLOC_MAX_BYTES)");
    int8_t *scratch = nullptr;
    if (operand_buffer(&scratch) != HATQ_OK)
        return hatq::report(HATQ_ERR_CUDA, "hatq_layer_noalloc: device address of the staging array unavailable");
    return hatq_layer(x, x_kind, s_in, n, h, w, L, y, scratch, (size_t)HATQ_NOALLOC_MAX_BYTES, stream);
}
