// noalloc.cu -- verify attention for callers that cannot allocate device
// memory.
//
// cs_verify_attention needs a caller-provided workspace.  Some callers have
// no way to provide one: code that runs under a host framework which owns
// every device allocation (its memory pool forbids a foreign cudaMalloc),
// serving loops that forbid any allocation after start-up because cudaMalloc
// can block the whole device for milliseconds, and thin language bindings
// that have no device allocator at all.  cs_verify_attention_noalloc runs the
// same kernel with its scratch in a fixed array compiled into this library.
//
// The array is a file-scope __device__ object of CS_NOALLOC_SCRATCH_BYTES:
// every GPU that loads the library holds that much memory until the process
// exits.  Host code cannot use the array's name as a device address (on the
// host the name is only a stand-in symbol), so the first call on each device
// looks the address up with cudaGetSymbolAddress while that device is
// current, and caches it.
#include <mutex>

#include "cs_internal.h"

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[CS_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
void* g_scratch_ptr[kMaxDevices] = {nullptr};
std::mutex g_scratch_mutex;

// Device address of the scratch array on the current device (set up once).
cs_status scratch_address(void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cs::cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices)
        return cs::fail(CS_ERR_UNSUPPORTED, "device ordinal %d is beyond %d", dev, kMaxDevices);
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    if (!g_scratch_ptr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return cs::cuda_fail(e, "cudaGetSymbolAddress(noalloc scratch)");
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return CS_OK;
}

}  // namespace

extern "C" cs_status cs_verify_attention_noalloc(const cs_attn_dims* dims, const void* q,
                                                 const void* k_pages, const void* v_pages,
                                                 const int32_t* page_table,
                                                 const int32_t* ctx_lens, int32_t n_draft,
                                                 void* out, cs_stream_t stream) {
    // The argument checks of cs_verify_attention, with the library's own
    // scratch standing in for the workspace.
    const size_t need = cs_verify_attention_workspace_bytes(dims, n_draft);
    if (need == 0) {
        // invalid dimensions: let the regular entry point report why
        return cs_verify_attention(dims, q, k_pages, v_pages, page_table, ctx_lens, n_draft, out,
                                   nullptr, 0, stream);
    }
    if (need > CS_NOALLOC_SCRATCH_BYTES)
        return cs::fail(CS_ERR_UNSUPPORTED,
                        "this problem needs %zu bytes of scratch; the allocation-free entry point "
                        "has %u bytes (use cs_verify_attention with a workspace)",
                        need, (unsigned)CS_NOALLOC_SCRATCH_BYTES);
    if (dims->batch == 0) return CS_OK;
    void* scratch = nullptr;
    cs_status st = scratch_address(&scratch);
    if (st != CS_OK) return st;
    // The status word must start at zero: clear it, so that a failed or
    // interrupted call cannot leak into this one.
    cudaError_t e = cudaMemsetAsync(scratch, 0, 256, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cs::cuda_fail(e, "cudaMemsetAsync(noalloc scratch)");
    return cs_verify_attention(dims, q, k_pages, v_pages, page_table, ctx_lens, n_draft, out,
                               scratch, CS_NOALLOC_SCRATCH_BYTES, stream);
}

// The status word at the start of the scratch array, read back for the
// caller (who never sees the array's address): the CS_DEVICE_* bits of the
// latest allocation-free call on this device.
extern "C" cs_status cs_verify_attention_noalloc_status(int32_t* status_out, cs_stream_t stream) {
    if (!status_out) return cs::fail(CS_ERR_INVALID_ARG, "status_out is NULL");
    void* scratch = nullptr;
    cs_status st = scratch_address(&scratch);
    if (st != CS_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemcpyAsync(status_out, scratch, sizeof(int32_t), cudaMemcpyDeviceToHost, s);
    if (e != cudaSuccess) return cs::cuda_fail(e, "cudaMemcpyAsync(noalloc status)");
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cs::cuda_fail(e, "cudaStreamSynchronize");
    return CS_OK;
}
