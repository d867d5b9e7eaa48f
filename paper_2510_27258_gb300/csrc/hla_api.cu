// C ABI of the HLA library: argument validation, workspace sizing, dispatch
// to the CUDA paths, error reporting.  See include/hla.h for the contract of
// every entry point.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include "hla_internal.h"

namespace hla {

static thread_local char g_last_error[512];

hla_status fail(hla_status st, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
    va_end(ap);
    return st;
}

void clear_last_error() { g_last_error[0] = 0; }

hla_status poll_header(void *header, cudaStream_t s) {
    WsHeader h{};
    hla_status st = cuda_status(cudaMemcpyAsync(&h, header, sizeof(h), cudaMemcpyDeviceToHost, s), "reading flag");
    if (st != HLA_OK) return st;
    st = cuda_status(cudaStreamSynchronize(s), "synchronising");
    if (st != HLA_OK) return st;
    if (h.error == kDevOk) return HLA_OK;
    st = cuda_status(cudaMemsetAsync(header, 0, sizeof(h), s), "clearing flag");
    if (st != HLA_OK) return st;
    return fail(HLA_ERR_TIMEOUT, "device-side wait gave up (where=%u detail=%u)", h.where, h.detail);
}

hla_status cuda_status(cudaError_t err, const char *what) {
    if (err == cudaSuccess) return HLA_OK;
    return fail(HLA_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(err), cudaGetErrorString(err));
}

namespace {

bool dim_ok(int x) { return x == 16 || x == 32 || x == 64 || x == 128; }

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t elem_bytes(hla_dtype dt) { return dt == HLA_BF16 ? 2 : 4; }

// Checks shared by the forward entry points; returns HLA_OK or the error.
hla_status check_forward(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int B, int H, int n,
                         int d, int dv, int masked, int normalized, float eps, int chunk, const float *state_in,
                         float *state_out) {
    if (dt != HLA_F32 && dt != HLA_BF16) return fail(HLA_ERR_INVALID_ARGUMENT, "unknown dtype %d", (int)dt);
    if (B < 0 || H < 0 || n < 0) return fail(HLA_ERR_INVALID_ARGUMENT, "negative size B=%d H=%d n=%d", B, H, n);
    if (d <= 0 || dv <= 0 || chunk <= 0)
        return fail(HLA_ERR_INVALID_ARGUMENT, "non-positive size d=%d dv=%d chunk=%d", d, dv, chunk);
    if ((masked != 0 && masked != 1) || (normalized != 0 && normalized != 1))
        return fail(HLA_ERR_INVALID_ARGUMENT, "flags must be 0 or 1 (masked=%d normalized=%d)", masked, normalized);
    if (!std::isfinite(eps)) return fail(HLA_ERR_INVALID_ARGUMENT, "eps must be finite");
    if (!dim_ok(d) || !dim_ok(dv))
        return fail(HLA_ERR_UNSUPPORTED, "d=%d dv=%d: supported sizes are 16, 32, 64, 128", d, dv);
    if (chunk > 128) return fail(HLA_ERR_UNSUPPORTED, "chunk=%d: supported chunks are 1..128", chunk);
    const long long tokens = (long long)B * H * n;
    if ((long long)B * H > (1LL << 31) - 1 || tokens * (d > dv ? d : dv) > (1LL << 40))
        return fail(HLA_ERR_UNSUPPORTED, "problem too large");
    if (tokens > 0 && (!q || !k || !v || !out))
        return fail(HLA_ERR_INVALID_ARGUMENT, "null q/k/v/out pointer");
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out) || !aligned16(state_in) ||
        !aligned16(state_out))
        return fail(HLA_ERR_INVALID_ARGUMENT, "q, k, v, out and states must be 16-byte aligned");
    (void)elem_bytes;
    return HLA_OK;
}

}  // namespace
}  // namespace hla

using namespace hla;

extern "C" {

const char *hla_status_string(hla_status status) {
    switch (status) {
        case HLA_OK: return "HLA_OK";
        case HLA_ERR_INVALID_ARGUMENT: return "HLA_ERR_INVALID_ARGUMENT";
        case HLA_ERR_UNSUPPORTED: return "HLA_ERR_UNSUPPORTED";
        case HLA_ERR_CUDA: return "HLA_ERR_CUDA";
        case HLA_ERR_TIMEOUT: return "HLA_ERR_TIMEOUT";
        case HLA_ERR_WORKSPACE: return "HLA_ERR_WORKSPACE";
    }
    return "HLA_ERR_UNKNOWN";
}

const char *hla_last_error(void) { return g_last_error; }

size_t hla2_state_floats(int d, int dv) {
    if (d <= 0 || dv <= 0) return 0;
    return (size_t)d * d + 2 * (size_t)d * dv + 2 * (size_t)d;
}

size_t hla3_state_floats(int d, int dv) {
    if (d <= 0 || dv <= 0) return 0;
    return 2 * (size_t)d * d + 4 * (size_t)d * dv + 4 * (size_t)d;
}

size_t hla2_workspace_bytes(int B, int H, int n, int d, int dv, int chunk, hla_dtype dt) {
    if (B < 0 || H < 0 || n < 0 || !dim_ok(d) || !dim_ok(dv) || chunk < 1 || chunk > 128) return 0;
    if (dt != HLA_F32 && dt != HLA_BF16) return 0;
    const int BH = B * H;
    size_t g = generic2_workspace_bytes(BH, n, d, dv, chunk);
    size_t f = fused2_workspace_bytes(BH, n, d, dv, chunk, dt, true);
    return align_up(g > f ? g : f, 256);
}

size_t hla3_workspace_bytes(int B, int H, int n, int d, int dv, int chunk, hla_dtype dt) {
    if (B < 0 || H < 0 || n < 0 || !dim_ok(d) || !dim_ok(dv) || chunk < 1 || chunk > 128) return 0;
    if (dt != HLA_F32 && dt != HLA_BF16) return 0;
    const int BH = B * H;
    const size_t g = generic3_workspace_bytes(BH, n, d, dv, chunk);
    const size_t c = chunked3_eligible(BH, n, d, dv, chunk) ? chunked3_workspace_bytes(BH, n, d, dv, chunk) : 0;
    const size_t t = hla3_tc_workspace_bytes(BH, n);
    const size_t gc = g > c ? g : c;
    return align_up(gc > t ? gc : t, 256);
}

hla_status hla2_forward(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int B, int H, int n,
                        int d, int dv, int masked, int normalized, float eps, int chunk, const float *state_in,
                        float *state_out, void *workspace, size_t workspace_bytes, hla_stream_t stream) {
    g_last_error[0] = 0;
    hla_status st = check_forward(q, k, v, out, dt, B, H, n, d, dv, masked, normalized, eps, chunk, state_in,
                                  state_out);
    if (st != HLA_OK) return st;
    const size_t need = hla2_workspace_bytes(B, H, n, d, dv, chunk, dt);
    if (!workspace || workspace_bytes < need)
        return fail(HLA_ERR_WORKSPACE, "workspace of %zu bytes needed, %zu given", need,
                    workspace ? workspace_bytes : (size_t)0);
    if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
        return fail(HLA_ERR_INVALID_ARGUMENT, "workspace must be 256-byte aligned");
    if ((long long)B * H == 0) return HLA_OK;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    st = cuda_status(cudaMemsetAsync(workspace, 0, kWsHeaderBytes, s), "clearing the workspace header");
    if (st != HLA_OK) return st;
    Fwd2 p{q, k, v, out, dt, B * H, n, d, dv, masked, normalized, eps, chunk, state_in, state_out,
           static_cast<char *>(workspace), workspace_bytes};
    if (fused2_applicable(p)) return cuda_status(fused2_forward(p, s), "fused forward");
    return cuda_status(generic2_forward(p, s), "generic forward");
}

int hla2_forward_path(int B, int H, int n, int d, int dv, int masked, int normalized, int chunk, hla_dtype dt,
                      int has_state_in, int has_state_out, int *launches) {
    const void *dummy = reinterpret_cast<const void *>(uintptr_t(256));
    if (check_forward(dummy, dummy, dummy, const_cast<void *>(dummy), dt, B, H, n, d, dv, masked, normalized, 0.f,
                      chunk, nullptr, nullptr) != HLA_OK)
        return -1;
    Fwd2 p{dummy, dummy, dummy, const_cast<void *>(dummy), dt, B * H, n, d, dv, masked, normalized, 0.f, chunk,
           has_state_in ? static_cast<const float *>(dummy) : nullptr,
           has_state_out ? static_cast<float *>(const_cast<void *>(dummy)) : nullptr, nullptr,
           hla2_workspace_bytes(B, H, n, d, dv, chunk, dt)};
    const bool fused = (long long)B * H > 0 && fused2_applicable(p);
    if (launches) {
        if ((long long)B * H == 0) *launches = 0;
        else if (fused) *launches = 1 + (has_state_in ? 1 : 0) + (has_state_out ? 2 : 0);
        else *launches = n > 0 ? 3 : 1;
    }
    return fused ? 1 : 0;
}

hla_status hla2_step(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int B, int H, int d,
                     int dv, int masked, int normalized, float eps, float *state, hla_stream_t stream) {
    g_last_error[0] = 0;
    hla_status st = check_forward(q, k, v, out, dt, B, H, 1, d, dv, masked, normalized, eps, 1, state, state);
    if (st != HLA_OK) return st;
    if ((long long)B * H > 0 && !state) return fail(HLA_ERR_INVALID_ARGUMENT, "null state pointer");
    if ((long long)B * H == 0) return HLA_OK;
    return cuda_status(step2_launch(q, k, v, out, dt, B * H, d, dv, masked, normalized, eps, state,
                                    reinterpret_cast<cudaStream_t>(stream)),
                       "decode step");
}

size_t hla2_sde_state_floats(int d, int dv) {
    if (d <= 0 || dv <= 0) return 0;
    return (size_t)d * d + (size_t)d * dv + (size_t)d;
}

hla_status hla2_state_to_sde(const float *state, float *sde, int B, int H, int d, int dv, hla_stream_t stream) {
    g_last_error[0] = 0;
    if (B < 0 || H < 0) return fail(HLA_ERR_INVALID_ARGUMENT, "negative size B=%d H=%d", B, H);
    if (!dim_ok(d) || !dim_ok(dv))
        return fail(HLA_ERR_UNSUPPORTED, "d=%d dv=%d: supported sizes are 16, 32, 64, 128", d, dv);
    const long long BH = (long long)B * H;
    if (BH == 0) return HLA_OK;
    if (BH > (1LL << 31) - 1) return fail(HLA_ERR_UNSUPPORTED, "problem too large");
    if (!state || !sde) return fail(HLA_ERR_INVALID_ARGUMENT, "null state pointer");
    if (!aligned16(state) || !aligned16(sde)) return fail(HLA_ERR_INVALID_ARGUMENT, "states must be 16-byte aligned");
    const uintptr_t a0 = reinterpret_cast<uintptr_t>(state), a1 = a0 + sizeof(float) * BH * hla2_state_floats(d, dv);
    const uintptr_t b0 = reinterpret_cast<uintptr_t>(sde), b1 = b0 + sizeof(float) * BH * hla2_sde_state_floats(d, dv);
    if (a0 < b1 && b0 < a1) return fail(HLA_ERR_INVALID_ARGUMENT, "state and sde must not overlap");
    return cuda_status(state_to_sde_launch(state, sde, (int)BH, d, dv, reinterpret_cast<cudaStream_t>(stream)),
                       "state conversion");
}

hla_status hla2_step_sde(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int B, int H, int d,
                         int dv, int normalized, float eps, float *sde, hla_stream_t stream) {
    g_last_error[0] = 0;
    hla_status st = check_forward(q, k, v, out, dt, B, H, 1, d, dv, 1, normalized, eps, 1, sde, sde);
    if (st != HLA_OK) return st;
    if ((long long)B * H == 0) return HLA_OK;
    if (!sde) return fail(HLA_ERR_INVALID_ARGUMENT, "null state pointer");
    return cuda_status(step2_sde_launch(q, k, v, out, dt, B * H, d, dv, normalized, eps, sde,
                                        reinterpret_cast<cudaStream_t>(stream)),
                       "decode step (S, D, e)");
}

size_t hla2_backward_workspace_bytes(int B, int H, int n, int d, int dv, int chunk, hla_dtype dt) {
    if (B < 0 || H < 0 || n < 0 || !dim_ok(d) || !dim_ok(dv) || chunk < 1 || chunk > 128) return 0;
    if (dt != HLA_F32 && dt != HLA_BF16) return 0;
    return align_up(backward2_workspace_bytes(B * H, n, d, dv, chunk), 256);
}

hla_status hla2_backward(const void *q, const void *k, const void *v, const void *dout, void *dq, void *dk, void *dv_,
                         hla_dtype dt, int B, int H, int n, int d, int dv, int normalized, float eps, int chunk,
                         void *workspace, size_t workspace_bytes, hla_stream_t stream) {
    g_last_error[0] = 0;
    hla_status st = check_forward(q, k, v, dv_, dt, B, H, n, d, dv, 1, normalized, eps, chunk, nullptr, nullptr);
    if (st != HLA_OK) return st;
    const long long tokens = (long long)B * H * n;
    if (tokens > 0 && (!dout || !dq || !dk)) return fail(HLA_ERR_INVALID_ARGUMENT, "null dout/dq/dk pointer");
    if (!aligned16(dout) || !aligned16(dq) || !aligned16(dk))
        return fail(HLA_ERR_INVALID_ARGUMENT, "dout, dq, dk and dv must be 16-byte aligned");
    const size_t need = hla2_backward_workspace_bytes(B, H, n, d, dv, chunk, dt);
    if (!workspace || workspace_bytes < need)
        return fail(HLA_ERR_WORKSPACE, "workspace of %zu bytes needed, %zu given", need,
                    workspace ? workspace_bytes : (size_t)0);
    if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
        return fail(HLA_ERR_INVALID_ARGUMENT, "workspace must be 256-byte aligned");
    if (tokens == 0) return HLA_OK;
    Bwd2 p{q, k, v, dout, dq, dk, dv_, dt, B * H, n, d, dv, normalized, eps, chunk, static_cast<char *>(workspace),
           workspace_bytes};
    return cuda_status(backward2_launch(p, reinterpret_cast<cudaStream_t>(stream)), "backward");
}

int hla2_backward_path(int B, int H, int n, int d, int dv, int normalized, int chunk, hla_dtype dt) {
    const void *dummy = reinterpret_cast<const void *>(uintptr_t(256));
    if (check_forward(dummy, dummy, dummy, const_cast<void *>(dummy), dt, B, H, n, d, dv, 1, normalized, 0.f, chunk,
                      nullptr, nullptr) != HLA_OK)
        return -1;
    Bwd2 p{dummy, dummy, dummy, dummy, const_cast<void *>(dummy), const_cast<void *>(dummy),
           const_cast<void *>(dummy), dt, B * H, n, d, dv, normalized, 0.f, chunk, nullptr,
           hla2_backward_workspace_bytes(B, H, n, d, dv, chunk, dt)};
    return ((long long)B * H > 0 && backward2_tc_applicable(p)) ? 1 : 0;
}

size_t ahla_state_floats(int d, int dv) {
    if (d <= 0 || dv <= 0) return 0;
    return 2 * (size_t)d * dv + 2 * (size_t)d;
}

size_t ahla_workspace_bytes(int B, int H, int n, int d, int dv, int chunk, hla_dtype dt) {
    if (B < 0 || H < 0 || n < 0 || !dim_ok(d) || !dim_ok(dv) || chunk < 1 || chunk > 128) return 0;
    if (dt != HLA_F32 && dt != HLA_BF16) return 0;
    return align_up(ahla_workspace_bytes_internal(B * H, n, d, dv, chunk), 256);
}

hla_status ahla_forward(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int B, int H, int n,
                        int d, int dv, int normalized, float eps, int chunk, const float *state_in, float *state_out,
                        void *workspace, size_t workspace_bytes, hla_stream_t stream) {
    g_last_error[0] = 0;
    hla_status st = check_forward(q, k, v, out, dt, B, H, n, d, dv, 1, normalized, eps, chunk, state_in, state_out);
    if (st != HLA_OK) return st;
    const size_t need = ahla_workspace_bytes(B, H, n, d, dv, chunk, dt);
    if (!workspace || workspace_bytes < need)
        return fail(HLA_ERR_WORKSPACE, "workspace of %zu bytes needed, %zu given", need,
                    workspace ? workspace_bytes : (size_t)0);
    if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
        return fail(HLA_ERR_INVALID_ARGUMENT, "workspace must be 256-byte aligned");
    if ((long long)B * H == 0) return HLA_OK;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    st = cuda_status(cudaMemsetAsync(workspace, 0, kWsHeaderBytes, s), "clearing the workspace header");
    if (st != HLA_OK) return st;
    Fwd2 p{q, k, v, out, dt, B * H, n, d, dv, 1, normalized, eps, chunk, state_in, state_out,
           static_cast<char *>(workspace), workspace_bytes};
    return cuda_status(ahla_forward_launch(p, s), "AHLA forward");
}

int ahla_forward_path(int B, int H, int n, int d, int dv, int normalized, int chunk, hla_dtype dt, int has_state_in,
                      int has_state_out) {
    const void *dummy = reinterpret_cast<const void *>(uintptr_t(256));
    if (check_forward(dummy, dummy, dummy, const_cast<void *>(dummy), dt, B, H, n, d, dv, 1, normalized, 0.f, chunk,
                      nullptr, nullptr) != HLA_OK)
        return -1;
    Fwd2 p{dummy, dummy, dummy, const_cast<void *>(dummy), dt, B * H, n, d, dv, 1, normalized, 0.f, chunk,
           has_state_in ? static_cast<const float *>(dummy) : nullptr,
           has_state_out ? static_cast<float *>(const_cast<void *>(dummy)) : nullptr, nullptr,
           ahla_workspace_bytes(B, H, n, d, dv, chunk, dt)};
    return ((long long)B * H > 0 && ahla_tc_applicable(p)) ? 1 : 0;
}

hla_status ahla_step(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int B, int H, int d,
                     int dv, int normalized, float eps, float *state, hla_stream_t stream) {
    g_last_error[0] = 0;
    hla_status st = check_forward(q, k, v, out, dt, B, H, 1, d, dv, 1, normalized, eps, 1, state, state);
    if (st != HLA_OK) return st;
    if ((long long)B * H == 0) return HLA_OK;
    if (!state) return fail(HLA_ERR_INVALID_ARGUMENT, "null state pointer");
    return cuda_status(ahla_step_launch(q, k, v, out, dt, B * H, d, dv, normalized, eps, state,
                                        reinterpret_cast<cudaStream_t>(stream)),
                       "AHLA decode step");
}

int hla3_forward_path(int B, int H, int n, int d, int dv, int masked, int normalized, int chunk, hla_dtype dt,
                      int has_state_in, int has_state_out, int *launches) {
    const void *dummy = reinterpret_cast<const void *>(uintptr_t(256));
    if (check_forward(dummy, dummy, dummy, const_cast<void *>(dummy), dt, B, H, n, d, dv, masked, normalized, 0.f,
                      chunk, nullptr, nullptr) != HLA_OK)
        return -1;
    Fwd2 p{dummy, dummy, dummy, const_cast<void *>(dummy), dt, B * H, n, d, dv, masked, normalized, 0.f, chunk,
           has_state_in ? static_cast<const float *>(dummy) : nullptr,
           has_state_out ? static_cast<float *>(const_cast<void *>(dummy)) : nullptr, nullptr,
           hla3_workspace_bytes(B, H, n, d, dv, chunk, dt)};
    int path = 0, nl = 0;
    if ((long long)B * H == 0) {
        path = 0;
    } else if (hla3_tc_applicable(p)) {
        path = 2;
        nl = hla3_tc_launches(B * H, n);
    } else if (!has_state_out && chunked3_eligible(B * H, n, d, dv, chunk)) {
        path = 1;
        nl = masked ? 5 + (has_state_in ? 1 : 0) : 3;
    } else {
        nl = 1;
    }
    if (launches) *launches = nl;
    return path;
}

hla_status hla3_forward(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int B, int H, int n,
                        int d, int dv, int masked, int normalized, float eps, int chunk, const float *state_in,
                        float *state_out, void *workspace, size_t workspace_bytes, hla_stream_t stream) {
    g_last_error[0] = 0;
    hla_status st = check_forward(q, k, v, out, dt, B, H, n, d, dv, masked, normalized, eps, chunk, state_in,
                                  state_out);
    if (st != HLA_OK) return st;
    const size_t need = hla3_workspace_bytes(B, H, n, d, dv, chunk, dt);
    if (!workspace || workspace_bytes < need)
        return fail(HLA_ERR_WORKSPACE, "workspace of %zu bytes needed, %zu given", need,
                    workspace ? workspace_bytes : (size_t)0);
    if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
        return fail(HLA_ERR_INVALID_ARGUMENT, "workspace must be 256-byte aligned");
    if ((long long)B * H == 0) return HLA_OK;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    st = cuda_status(cudaMemsetAsync(workspace, 0, kWsHeaderBytes, s), "clearing the workspace header");
    if (st != HLA_OK) return st;
    Fwd2 p{q, k, v, out, dt, B * H, n, d, dv, masked, normalized, eps, chunk, state_in, state_out,
           static_cast<char *>(workspace), workspace_bytes};
    if (hla3_tc_applicable(p)) return cuda_status(hla3_tc_forward(p, s), "third-order forward (tensor cores)");
    // chunk-parallel unless the final state is wanted (the serial kernel also carries G1..G3, h1..h3)
    if (!state_out && chunked3_eligible(B * H, n, d, dv, chunk))
        return cuda_status(chunked3_forward(p, s), "third-order forward (chunked)");
    return cuda_status(generic3_forward(p, s), "third-order forward");
}

hla_status hla_poll_error(void *workspace, hla_stream_t stream) {
    g_last_error[0] = 0;
    if (!workspace) return fail(HLA_ERR_INVALID_ARGUMENT, "null workspace");
    return poll_header(workspace, reinterpret_cast<cudaStream_t>(stream));
}

}  // extern "C"
