// ts_router.cu -- MoE router (Sec. 4): logits r = W_r x, top-k experts (a
// lower expert index wins a tie), softmax over the k picked logits.
// One CTA per token; warp e computes logit e with 16-byte streaming loads.
// In stack mode the CTA first normalises its residual row (the stack glue)
// and publishes the activations for the grouped expert kernels.
#include "ts_kernels.cuh"

namespace tsffn {

template <typename T>
__global__ void __launch_bounds__(256) k_router(const RouterLaunch a) {
    constexpr int VEC = Vec<T>::N;
    extern __shared__ __align__(16) float xs[];  // [d]
    __shared__ float logit[kMaxExperts];
    __shared__ float red[8];
    const int t = blockIdx.x;
    const int d = a.d;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;

    pdl_wait();
    pdl_launch_dependents();
    if (a.h != nullptr) {
        block_rmsnorm<T>(a.h + (size_t)t * d, d, xs, red);
        for (int i = threadIdx.x; i < d; i += blockDim.x)
            Vec<T>::store1(a.xbuf, (size_t)t * d + i, xs[i]);
    } else {
        for (int i = threadIdx.x; i < d; i += blockDim.x)
            xs[i] = Vec<T>::load1(a.x, (size_t)t * d + i);
    }
    __syncthreads();

    for (int e = warp; e < a.n_experts; e += nw) {
        const T* row = static_cast<const T*>(a.wr) + (size_t)e * d;
        float acc = 0.0f;
        for (int col = lane * VEC; col < d; col += kWarp * VEC) {
            float f[VEC];
            Vec<T>::unpack(ld_stream(row + col), f);
#pragma unroll
            for (int q = 0; q < VEC; ++q) acc = fmaf(f[q], xs[col + q], acc);
        }
        acc = warp_sum(acc);
        if (lane == 0) logit[e] = acc;
    }
    __syncthreads();

    if (threadIdx.x == 0) {
        TokenRoute r;
        unsigned taken = 0u;
        for (int k = 0; k < kMaxTopK; ++k) {
            r.sel[k] = -1;
            r.w[k] = 0.0f;
        }
        for (int k = 0; k < a.top_k; ++k) {
            int best = -1;
            for (int e = 0; e < a.n_experts; ++e) {
                if ((taken >> e) & 1u) continue;
                if (best < 0 || logit[e] > logit[best]) best = e;
            }
            r.sel[k] = best;
            taken |= 1u << best;
        }
        float z = 0.0f;
        for (int k = 0; k < a.top_k; ++k) z += expf(logit[r.sel[k]] - logit[r.sel[0]]);
        for (int k = 0; k < a.top_k; ++k) r.w[k] = expf(logit[r.sel[k]] - logit[r.sel[0]]) / z;
        a.route[t] = r;
    }
}

cudaError_t launch_router(const RouterLaunch& a, int wdtype, cudaStream_t stream, bool pdl) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.batch);
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = (size_t)a.d * sizeof(float);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    if (wdtype == 1) return cudaLaunchKernelEx(&cfg, k_router<__nv_bfloat16>, a);
    return cudaLaunchKernelEx(&cfg, k_router<float>, a);
}

cudaError_t prepare_router() {
    cudaError_t e = cudaFuncSetAttribute(k_router<__nv_bfloat16>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, kRouterMaxD * 4);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_router<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kRouterMaxD * 4);
    return e;
}

}  // namespace tsffn
