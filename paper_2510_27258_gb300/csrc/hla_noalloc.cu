// hla2_forward_noalloc: the fused second-order forward for callers that cannot
// allocate device memory (see include/hla.h).  Its scratch is a fixed array in
// device memory that belongs to this library, not a caller-provided workspace.
#include <cmath>
#include <mutex>

#include "hla_internal.h"

namespace hla {
namespace {

// Maximum scratch of one call.  Every GPU on which the library runs holds this
// array until the process exits.
constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
void *g_scratch_ptr[kMaxDevices] = {};  // device address of the array, per device

// Device address of the scratch array on the current device (first use on a
// device looks it up with cudaGetSymbolAddress while that device is current).
hla_status scratch_address(void **out) {
    int dev = 0;
    hla_status st = cuda_status(cudaGetDevice(&dev), "cudaGetDevice");
    if (st != HLA_OK) return st;
    if (dev < 0 || dev >= kMaxDevices) return fail(HLA_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        st = cuda_status(cudaGetSymbolAddress(&p, g_noalloc_scratch), "cudaGetSymbolAddress(scratch)");
        if (st != HLA_OK) return st;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return HLA_OK;
}

}  // namespace
}  // namespace hla

using namespace hla;

extern "C" hla_status hla2_forward_noalloc(const void *q, const void *k, const void *v, void *out, hla_dtype dt,
                                           int B, int H, int n, int d, int dv, int masked, int normalized,
                                           float eps, int chunk, const float *state_in, hla_stream_t stream) {
    // Same argument checks as hla2_forward; only the fused path is offered.
    clear_last_error();
    int launches = 0;
    const int path = hla2_forward_path(B, H, n, d, dv, masked, normalized, chunk, dt, state_in != nullptr, 0,
                                       &launches);
    if (path < 0) return fail(HLA_ERR_UNSUPPORTED, "arguments not supported by hla2_forward");
    if ((long long)B * H == 0 || n == 0) return HLA_OK;  // nothing to compute (no final state is written)
    if (path != 1)
        return fail(HLA_ERR_UNSUPPORTED,
                    "hla2_forward_noalloc serves the fused path only (bf16, d and dv in {64, 128}, masked, no "
                    "state_out; an initial state only with d = dv = 128; sm_103)");
    if (!q || !k || !v || !out) return fail(HLA_ERR_INVALID_ARGUMENT, "null q/k/v/out pointer");
    const uintptr_t mis = (reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(k) |
                           reinterpret_cast<uintptr_t>(v) | reinterpret_cast<uintptr_t>(out) |
                           reinterpret_cast<uintptr_t>(state_in)) & 15u;
    if (mis) return fail(HLA_ERR_INVALID_ARGUMENT, "q, k, v, out and state_in must be 16-byte aligned");
    if (!std::isfinite(eps)) return fail(HLA_ERR_INVALID_ARGUMENT, "eps must be finite");
    const size_t need = fused2_workspace_bytes(B * H, n, d, dv, chunk, dt, false);
    if (need > kNoAllocScratchBytes)
        return fail(HLA_ERR_WORKSPACE, "these sizes need %zu bytes of scratch; hla2_forward_noalloc has %zu", need,
                    kNoAllocScratchBytes);
    void *scratch = nullptr;
    hla_status st = scratch_address(&scratch);
    if (st != HLA_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    // the error word must start at zero; the fused launch clears its own counters
    st = cuda_status(cudaMemsetAsync(scratch, 0, kWsHeaderBytes, s), "clearing the scratch header");
    if (st != HLA_OK) return st;
    Fwd2 p{q, k, v, out, dt, B * H, n, d, dv, masked, normalized, eps, chunk, state_in, nullptr,
           static_cast<char *>(scratch), kNoAllocScratchBytes};
    return cuda_status(fused2_forward(p, s), "fused forward (no-alloc)");
}

extern "C" hla_status hla_poll_error_noalloc(hla_stream_t stream) {
    clear_last_error();
    void *scratch = nullptr;
    hla_status st = scratch_address(&scratch);
    if (st != HLA_OK) return st;
    return poll_header(scratch, reinterpret_cast<cudaStream_t>(stream));
}
