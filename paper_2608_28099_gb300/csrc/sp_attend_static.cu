// sp_attend_static: the attention step without any device allocation.
//
// sp_attend needs a caller-allocated workspace for its split-KV partials.
// Some callers cannot allocate device memory at the point where they
// classify: a monitor running on the decoding hot path must not call
// cudaMalloc, because cudaMalloc can synchronise the device and stall the
// decoding stream it is meant to leave undisturbed; and serving frameworks that
// hand all device memory to their own pool allocator leave a library no way to
// obtain any.  This entry point takes the scratch from a fixed array in the
// library's own device memory instead, so the caller passes only inputs and
// outputs.
//
// The array is a file-scope __device__ object of kStaticScratchBytes; every
// GPU that loads the library holds it until the process exits.  Host code
// cannot use the array's name as a device address, so the first call on each
// device looks the address up with cudaGetSymbolAddress (with that device
// current) and caches it.  Under CUDA's lazy module loading that first call
// also loads this file's module, which is when the array's memory is committed
// on the device (an allocation, and possibly a synchronisation): make the first
// call on each device at set-up time, before any stream capture and before the
// decoding loop it must not disturb.  The cached address belongs to the
// device's primary context; it is not valid across cudaDeviceReset.
// All calls share the one array: calls whose work overlaps on the GPU (other
// streams, other host threads) race on it and must be serialised by the
// caller.  Nothing in it needs to start at zero: every partial the merge reads
// is written earlier in the same call.
#include <stdio.h>

#include <mutex>

#include "sp_common.cuh"

namespace {

constexpr size_t kStaticScratchBytes = 32u << 20;  // 32 MiB
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

std::mutex g_lock;
void *g_scratch_ptr[kMaxDevices] = {};

thread_local char g_msg[256];

// Device address of g_static_scratch on the current device (looked up once).
cudaError_t scratch_address(void **out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> guard(g_lock);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_static_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return cudaSuccess;
}

}  // namespace

extern "C" {

sp_status sp_attend_static(sp_stream stream, const sp_attn_dims *dims, int batch,
                           const int *d_seq_ids, const int *d_seq_lens, const sp_kv_cache *kv,
                           const float *d_q, const float *d_k_new, const float *d_v_new,
                           void *d_out, int out_dtype, int *d_status, int *d_gathered_pages) {
    const size_t need = sp_attend_workspace_bytes(dims, batch);
    if (need == 0) {
        snprintf(g_msg, sizeof g_msg,
                 "sp_attend_static: invalid attention dims or batch (heads, k_rows, "
                 "max_seq_len or split_tokens out of range)");
        sp::set_error_text(g_msg);
        return SP_ERR_INVALID_ARG;
    }
    if (need > kStaticScratchBytes) {
        snprintf(g_msg, sizeof g_msg,
                 "sp_attend_static: this batch needs %zu bytes of scratch, more than the "
                 "%zu-byte static array; use sp_attend with a workspace",
                 need, kStaticScratchBytes);
        sp::set_error_text(g_msg);
        return SP_ERR_INVALID_ARG;
    }
    void *scratch = nullptr;
    cudaError_t e = scratch_address(&scratch);
    if (e != cudaSuccess) {
        snprintf(g_msg, sizeof g_msg, "sp_attend_static: cudaGetSymbolAddress failed: %s",
                 cudaGetErrorString(e));
        sp::set_error_text(g_msg);
        return SP_ERR_CUDA;
    }
    return sp_attend(stream, dims, batch, d_seq_ids, d_seq_lens, kv, d_q, d_k_new, d_v_new, d_out,
                     out_dtype, scratch, kStaticScratchBytes, d_status, d_gathered_pages);
}

}  // extern "C"
