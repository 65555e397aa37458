// ts_predict.h -- launch parameters of the activation predictor (Sec. 7):
// a two-layer ReLU MLP scores every neuron for each token, a neuron's key over
// the batch is its largest score, and the K best keys (a lower neuron index
// winning a tie) form an ascending list that drives the predictor mode of the
// FFN kernels.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace tsffn {

constexpr int kPredMaxBatch = 8;   // tokens per prediction (x rows held in shared memory)
constexpr int kPredMaxSplits = 8;  // K-splits of a W1 row
constexpr int kPredHistBins = 4096;  // histogram of the keys' top 12 bits
constexpr int kPredHistParts = 8;    // copies of it, by score CTA, to spread the atomics

struct PredictLaunch {
    int d, r, m, batch;
    const void* x;       // [batch][d] activations (weight dtype), or nullptr with h
    const float* h;      // [batch][d] fp32 residual: x = rmsnorm(h) (stack mode)
    const void* w1;      // [r][d] first layer
    const void* w2;      // [m][r] second layer
    float* hid;          // [splits][batch][r] partial pre-activations of the hidden layer
    int splits;          // W1 rows are summed in `splits` contiguous segments
    int hid_grid;        // CTAs of the hidden-layer kernel
    int score_grid;      // CTAs of the score kernel
    unsigned* key;       // [m] order-preserving bits of max_t s[t][j]
    unsigned* hist;      // [kPredHistParts][kPredHistBins] count of keys per top-12-bit value, one
                         // copy per score-CTA residue mod kPredHistParts (cleared by the
                         // hidden-layer kernel, filled by the score kernel, summed by the select)
    float* scores;       // [batch][m] fp32 scores, or nullptr
    int K;               // list length, 1 <= K <= m
    int32_t* list;       // [K] out: ascending neuron ids
};

// Whether (d, r) with this element size has a kernel; the hidden layer's x
// rows must fit in `optin_smem` bytes of shared memory.
bool predict_supported(int elem_bytes, int d, int r, int batch, int optin_smem);
// Split count and grids for a device with `num_sms` SMs.
void predict_geometry(PredictLaunch* p, int elem_bytes, int num_sms);
cudaError_t prepare_predict(int optin_smem);
// Hidden layer, scores and list selection: three launches on `stream`.
cudaError_t launch_predict(const PredictLaunch& p, int elem_bytes, cudaStream_t stream, bool pdl);

}  // namespace tsffn
