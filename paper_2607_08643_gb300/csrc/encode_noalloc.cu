// encode_noalloc.cu -- bisco_encode_noalloc: the offline encoder with its
// scratch memory taken from a fixed array that lives inside this library,
// for callers that cannot allocate device memory themselves (for example a
// host application whose own allocator has reserved the device memory and
// forbids other cudaMalloc calls, or code that must avoid the device-wide
// synchronisation cudaMalloc/cudaFree can cause).
//
// The array is a file-scope __device__ object: every GPU that loads the
// library holds it (BISCO_ENCODE_NOALLOC_MAX_K * 13 bytes) until the process
// exits.  Host code cannot use the array's name as a device address, so the
// first call on each device looks the address up with cudaGetSymbolAddress
// while that device is current; make that first call before any stream
// capture.  All calls share the one array: calls that overlap on the GPU
// (two streams, or two host threads) race on it and must be serialised by
// the caller.  Each call writes every scratch entry it later reads, so
// nothing left from an earlier call needs clearing.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "bisco_host.h"

namespace bisco {
namespace {

// scores (8 B), ranks (4 B) and the protected map (1 B) per input column,
// each region rounded to 256 B: 13 bytes per column for K a multiple of 256.
constexpr size_t kNoallocScratchBytes = static_cast<size_t>(BISCO_ENCODE_NOALLOC_MAX_K) * 13;
static_assert(BISCO_ENCODE_NOALLOC_MAX_K % 256 == 0, "max K must be a multiple of 256");

static __device__ __align__(256) unsigned char g_encode_scratch[kNoallocScratchBytes];

constexpr int kMaxDev = 64;
std::mutex g_scratch_mu;
void *g_scratch_ptr[kMaxDev] = {};

// Device address of the scratch array on the current device (looked up once
// per device).
bisco_status scratch_address(void **out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return BISCO_ERR_CUDA;
    std::lock_guard<std::mutex> lk(g_scratch_mu);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_encode_scratch) != cudaSuccess || !p) return BISCO_ERR_CUDA;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return BISCO_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace bisco

extern "C" bisco_status bisco_encode_noalloc(const uint16_t *W_bf16, const float *g,
                                             const bisco_layer *L, bisco_stream_t stream) {
    using namespace bisco;
    bisco_status st = check_layer(L, true);   // the same checks as bisco_encode
    if (st != BISCO_OK) return st;
    if (!W_bf16 || !aligned16(W_bf16) || (g && (reinterpret_cast<uintptr_t>(g) & 3u)))
        return BISCO_ERR_INVALID_ARG;
    // What this entry point leaves out: output-row protection, payloads
    // other than INT8, and K beyond the array.
    if (L->protect_axis != 0 || L->protect_format != BISCO_PROT_INT8) return BISCO_ERR_UNSUPPORTED;
    if (L->k_in > BISCO_ENCODE_NOALLOC_MAX_K) return BISCO_ERR_UNSUPPORTED;
    if (encode_workspace_bytes(L->n_out, L->k_in) > kNoallocScratchBytes) return BISCO_ERR_UNSUPPORTED;
    void *scratch = nullptr;
    st = scratch_address(&scratch);
    if (st != BISCO_OK) return st;
    int *err = device_error_word(&st);
    if (!err) return st;
    return launch_encode(W_bf16, g, *L, scratch, err, reinterpret_cast<cudaStream_t>(stream));
}
