// Split-K decode attention for callers that cannot allocate device memory.
//
// ee_attention_decode needs a caller-provided scratch buffer for its per-split
// partial results and arrival counters.  Some callers have no way to provide
// one: their device memory is owned entirely by another allocator (a serving
// framework's pool that has reserved almost all of HBM, where an extra
// cudaMalloc fails or fragments the pool), they run on latency-critical paths
// where cudaMalloc/cudaFree may synchronise the device and stall other work,
// or they are plugins with no allocator handed to them.  For them,
// ee_attention_decode_static keeps its scratch in a fixed area of device
// memory that is part of this library's image: every GPU that loads the
// library holds EE_STATIC_ATTN_SCRATCH_BYTES for it until the process exits.
#include <cuda_runtime.h>

#include <string>

#include "ee.h"
#include "ee_internal.h"

namespace {

constexpr size_t kStaticBytes = EE_STATIC_ATTN_SCRATCH_BYTES;
constexpr size_t kAlign = 256;

// The shared scratch area.  Host code only ever sees a stand-in for this
// symbol: its device address comes from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_attn_scratch[kStaticBytes];

size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// Device address of the scratch area on the current device.  It is looked
// up on every call: once the library's device code is loaded on a device the
// lookup is a host-side table read, and an address kept from an earlier call
// would go stale if the caller reset the device (cudaDeviceReset), after
// which the code, and the area with it, may load at another address.  The
// first call on a device loads the code there.
int scratch_address(void** out) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_attn_scratch);
    if (e != cudaSuccess || !p)
        return ee::set_last_error(EE_ECUDA, (std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e)).c_str());
    *out = p;
    return EE_OK;
}

}  // namespace

extern "C" int ee_attention_decode_static(const float* q, const uint16_t* k_pages, const uint16_t* v_pages,
                                          const int32_t* page_table, int T, int n_heads, int n_kv_heads,
                                          int head_dim, int page_size, float* out, void* stream) {
    if (!q || !k_pages || !v_pages || !page_table || !out) return ee::set_last_error(EE_EINVAL, "NULL argument");
    if (n_heads <= 0 || n_kv_heads <= 0 || (head_dim != 64 && head_dim != 128))
        return ee::set_last_error(EE_EINVAL, "bad shape: head_dim must be 64 or 128");
    if (n_heads % n_kv_heads || n_heads / n_kv_heads > 8)
        return ee::set_last_error(EE_EINVAL, "bad head grouping");
    if (T <= 0 || page_size <= 0) return ee::set_last_error(EE_EINVAL, "T and page_size must be positive");
    const size_t part = align_up(4 * (size_t)n_heads * ee::kAttnMaxSplits * (head_dim + 2));
    const size_t need = part + 4 * (size_t)n_kv_heads;
    if (need > kStaticBytes) {
        const std::string m = "this shape needs " + std::to_string(need) + " bytes of scratch but the static area holds " +
                              std::to_string(kStaticBytes) + " (n_heads * (head_dim + 2) must be at most " +
                              std::to_string((kStaticBytes - 4 * (size_t)n_kv_heads) / (4 * ee::kAttnMaxSplits)) + ")";
        return ee::set_last_error(EE_EINVAL, m.c_str());
    }
    void* base = nullptr;
    int rc = scratch_address(&base);
    if (rc != EE_OK) return rc;
    cudaStream_t s = (cudaStream_t)stream;
    char* sc = (char*)base;
    ee::AttnArgs a{};
    a.q = q;
    a.kp = k_pages;
    a.vp = v_pages;
    a.page_table = page_table;
    a.ctl = nullptr;
    a.T = T;
    a.A = n_heads;
    a.KH = n_kv_heads;
    a.page_size = page_size;
    a.out = out;
    a.part = (float*)sc;
    a.ticket = (int*)(sc + part);
    // The arrival counters must start at zero; the partial sums need no clearing.
    cudaError_t e = cudaMemsetAsync(a.ticket, 0, 4 * (size_t)n_kv_heads, s);
    if (e == cudaSuccess) e = ee::launch_attention(a, head_dim, false, s);
    if (e != cudaSuccess) return ee::set_last_error(EE_ECUDA, cudaGetErrorString(e));
    return EE_OK;
}
