// Internal declarations of the HLA CUDA library (not part of the public ABI).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "hla.h"

namespace hla {

// ---------------------------------------------------------------------------
// Workspace: the first kWsHeaderBytes bytes of every workspace hold the
// device-side error word (read by hla_poll_error); scratch follows.
// ---------------------------------------------------------------------------
constexpr size_t kWsHeaderBytes = 256;

struct WsHeader {
    unsigned int error;   // 0 = ok, otherwise a DevError code
    unsigned int where;   // kernel-specific location of the failure
    unsigned int detail;  // kernel-specific detail (e.g. a chunk index)
};

enum DevError : unsigned int { kDevOk = 0, kDevTimeout = 1 };

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Records a host-side error message for hla_last_error() and returns `st`.
hla_status fail(hla_status st, const char *fmt, ...);
// Empties the message hla_last_error() returns (every entry point starts with it).
void clear_last_error();
// Reads the device-side error word of a workspace header (waiting for `stream`),
// clears it, and maps it to HLA_OK / HLA_ERR_TIMEOUT (HLA_ERR_CUDA if a call fails).
hla_status poll_header(void *header, cudaStream_t stream);
// Maps a CUDA error to HLA_ERR_CUDA (recording the CUDA message), or HLA_OK.
hla_status cuda_status(cudaError_t err, const char *what);

// ---------------------------------------------------------------------------
// token element access
// ---------------------------------------------------------------------------
__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }
__device__ __forceinline__ void from_f32(float *p, float x) { *p = x; }
__device__ __forceinline__ void from_f32(__nv_bfloat16 *p, float x) { *p = __float2bfloat16_rn(x); }

// ---------------------------------------------------------------------------
// forward problem description shared by the forward paths
// ---------------------------------------------------------------------------
struct Fwd2 {
    const void *q, *k, *v;
    void *out;
    hla_dtype dt;
    int BH, n, d, dv, masked, normalized;
    float eps;
    int chunk;
    const float *state_in;
    float *state_out;
    char *ws;        // workspace base (header included)
    size_t ws_bytes;
};

// generic fp32 SIMT path (any supported shape)
size_t generic2_workspace_bytes(int BH, int n, int d, int dv, int chunk);
cudaError_t generic2_forward(const Fwd2 &p, cudaStream_t stream);

// fused tcgen05 path (bf16, d = dv in {64, 128}); returns false if it does not apply
size_t fused2_workspace_bytes(int BH, int n, int d, int dv, int chunk, hla_dtype dt, bool with_state);
bool fused2_applicable(const Fwd2 &p);
cudaError_t fused2_forward(const Fwd2 &p, cudaStream_t stream);

// decode step
cudaError_t step2_launch(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int BH, int d,
                         int dv, int masked, int normalized, float eps, float *state, cudaStream_t stream);

// decode step on the (S, D, e) state, and the conversion of paper tuples to it
cudaError_t step2_sde_launch(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int BH, int d,
                             int dv, int normalized, float eps, float *state, cudaStream_t stream);
cudaError_t state_to_sde_launch(const float *src, float *dst, int BH, int d, int dv, cudaStream_t stream);

// gradients of masked second order (reverse chunk scan)
struct Bwd2 {
    const void *q, *k, *v, *dout;
    void *dq, *dk, *dval;
    hla_dtype dt;
    int BH, n, d, dv, normalized;
    float eps;
    int chunk;
    char *ws;
    size_t ws_bytes;
};
size_t backward2_workspace_bytes(int BH, int n, int d, int dv, int chunk);
cudaError_t backward2_launch(const Bwd2 &p, cudaStream_t stream);
// the backward on the tensor cores (hla_backward_sm103.cu): bf16, d = dv = 64, plain output
size_t backward2_tc_workspace_bytes(int BH, int n);
bool backward2_tc_applicable(const Bwd2 &p);
cudaError_t backward2_tc_launch(const Bwd2 &p, cudaStream_t stream);

// AHLA (asymmetric second order): chunk-parallel forward and decode step
size_t ahla_workspace_bytes_internal(int BH, int n, int d, int dv, int chunk);
// tensor-core AHLA forward (bf16, d and dv in {64, 128}, plain output, no states, sm_103)
bool ahla_tc_applicable(const Fwd2 &p);
cudaError_t ahla_tc_forward(const Fwd2 &p, cudaStream_t stream);
cudaError_t ahla_forward_launch(const Fwd2 &p, cudaStream_t stream);
cudaError_t ahla_step_launch(const void *q, const void *k, const void *v, void *out, hla_dtype dt, int BH, int d,
                             int dv, int normalized, float eps, float *state, cudaStream_t stream);

// third order
size_t generic3_workspace_bytes(int BH, int n, int d, int dv, int chunk);
cudaError_t generic3_forward(const Fwd2 &p, cudaStream_t stream);
// chunk-parallel third order (no state_out)
size_t chunked3_workspace_bytes(int BH, int n, int d, int dv, int chunk);
bool chunked3_eligible(int BH, int n, int d, int dv, int chunk);
cudaError_t chunked3_forward(const Fwd2 &p, cudaStream_t stream);

// Masked third-order forward on the tensor cores (hla3_sm103.cu): fp32, d = dv = 32,
// plain output, no states
size_t hla3_tc_workspace_bytes(int BH, int n);
bool hla3_tc_applicable(const Fwd2 &p);
int hla3_tc_launches(int BH, int n);
cudaError_t hla3_tc_forward(const Fwd2 &p, cudaStream_t stream);

}  // namespace hla
