// ts_wide.h -- launch block of the wide-pass kernels (ts_wide.cu): passes of
// 9-64 tokens of a bf16 FFN as gathered tensor-core GEMMs.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace tsffn {

struct WideLaunch {
    int d, m, n_rows, batch;      // batch: 9 .. 64 tokens
    const int32_t* rows;          // predictor list (ascending neuron ids) or nullptr
    const __nv_bfloat16* x;       // [batch][d] activations
    const __nv_bfloat16* wg;      // [m][d]
    const __nv_bfloat16* wu;
    const __nv_bfloat16* wd;
    float* gval;                  // [batch][n_rows] gate pre-activations
    __nv_bfloat16* c_hi;          // [n_rows][64] c = g u at both-active rows, hi part
    __nv_bfloat16* c_lo;          // [n_rows][64] lo part (c - hi)
    float* partial;               // [ks][batch][d] down projection per slice of the active rows
    int ks;                       // slices
    uint8_t* gbits;               // [batch][nbytes] gate-active bitmaps (per row-space position)
    uint8_t* bbits;               // [batch][nbytes] both-active bitmaps
    uint8_t* ubits;               // [nbytes] union both-active
    uint8_t* ugbits;              // [nbytes] union gate-active
    int nbytes;                   // bitmap bytes per token (multiple of 4)
    unsigned* status;
    float* y;                     // [batch][d] output, or
    float* h;                     // [batch][d] residual: h += y (residual_out)
    int residual_out;
};

// Whether a pass of `batch` tokens takes the wide kernels.
bool wide_supported(int wdtype, int d, int m, int batch);
// Slices of the active rows for the down projection (one CTA per slice and 256 columns).
int wide_slices(int d, int num_sms);
cudaError_t prepare_wide();
// gate, up, down and the reduction of one pass (programmatic dependent launch
// between them; `pdl` for the first).
cudaError_t launch_wide(const WideLaunch& L, cudaStream_t stream, bool pdl);
// x = rmsnorm(h) with x[d-1] = 1, bf16, for the stack.
cudaError_t launch_wide_norm(const WideLaunch& L, const float* h, __nv_bfloat16* xout, cudaStream_t stream,
                             bool pdl);

}  // namespace tsffn
