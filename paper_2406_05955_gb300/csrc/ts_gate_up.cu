// ts_gate_up.cu -- fused gate GEMV + ReLU + compaction and gathered up
// projection + dReLU product + second compaction (Eq. 1 with Eq. 2).
//
// Work item = (expert, chunk of kChunk consecutive rows of the row space).
// One warp owns an item end to end, so no block-level barrier sits in the
// streaming loop:
//   1. g = W_gate[j] . x for the chunk's rows and every token of the item;
//   2. ballot(any token has g > 0) -> the chunk's gate-active rows;
//   3. u = W_up[j] . x only for those rows (the W_up bytes the method saves);
//   4. ballot(g > 0 and u > 0) per token -> one bitmap byte per chunk per
//      token plus the union byte, and c = w_route * g * u for union rows.
// Rows stream with 16-byte ld.global.nc.L1::no_allocate loads, R rows at a
// time so each activation element read from shared memory feeds R rows.
// The activations sit in shared memory as fp32 (the bf16 values exactly).
#include "ts_kernels.cuh"

namespace tsffn {

// Rows per dot-product group and 16-byte loads per lane per row per step,
// chosen so a warp keeps about 8 KB of weights in flight and the
// accumulators stay in registers.
template <typename T, int NT>
struct GateUpShape {
    static constexpr int R = NT == 1 ? 1 : (NT == 2 ? 4 : (NT == 4 ? 2 : 1));
    static constexpr int U = (sizeof(T) == 2 ? 16 : 8) / R;  // R <= 8, so U >= 1
};

// acc[r][k] = sum_i W[row[r]][i] * xs[xo[k] + i] for k < ntok; rows with
// row[r] < 0 give 0. Every lane ends with the full sums.
template <typename T, int NT, int R, int U>
__device__ __forceinline__ void rows_dot(const T* __restrict__ W, const int (&row)[R], int d,
                                         const float* __restrict__ xs, const int (&xo)[NT],
                                         int ntok, int lane, float (&acc)[R][NT]) {
    constexpr int VEC = Vec<T>::N;
    constexpr int STEP = kWarp * VEC;
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
        for (int k = 0; k < NT; ++k) acc[r][k] = 0.0f;

    for (int base = lane * VEC; base < d; base += STEP * U) {
        uint4 v[R][U];
#pragma unroll
        for (int r = 0; r < R; ++r)
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int col = base + u * STEP;
                if (row[r] >= 0 && col < d)
                    v[r][u] = ld_stream(W + (size_t)row[r] * (size_t)d + col);
                else
                    v[r][u] = make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int col = base + u * STEP;
            if (col < d) {
                float f[R][VEC];
#pragma unroll
                for (int r = 0; r < R; ++r) Vec<T>::unpack(v[r][u], f[r]);
#pragma unroll
                for (int k = 0; k < NT; ++k) {
                    if (k < ntok) {
#pragma unroll
                        for (int q = 0; q < VEC; q += 4) {
                            const float4 xv = *reinterpret_cast<const float4*>(xs + xo[k] + col + q);
#pragma unroll
                            for (int r = 0; r < R; ++r) {
                                float a = acc[r][k];
                                a = fmaf(f[r][q + 0], xv.x, a);
                                a = fmaf(f[r][q + 1], xv.y, a);
                                a = fmaf(f[r][q + 2], xv.z, a);
                                a = fmaf(f[r][q + 3], xv.w, a);
                                acc[r][k] = a;
                            }
                        }
                    }
                }
            }
        }
    }
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
        for (int k = 0; k < NT; ++k) acc[r][k] = warp_sum(acc[r][k]);
}

template <typename T, int NT>
__global__ void __launch_bounds__(kGateUpWarps * kWarp, 2)
k_gate_up(const FfnLaunch a, int prefetch_rows) {
    using S = GateUpShape<T, NT>;
    constexpr int R = S::R;
    constexpr int U = S::U;
    extern __shared__ __align__(16) float xs[];  // [tokens][d] fp32
    __shared__ ExpertSets es;
    __shared__ float red[kGateUpWarps];

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int d = a.d;
    const int n_chunks = (a.n_rows + kChunk - 1) / kChunk;
    const int gwarp = blockIdx.x * kGateUpWarps + warp;
    const int nwarps = gridDim.x * kGateUpWarps;

    // Weights never change, so their first rows may be pulled into L2 while
    // the previous kernel on the stream is still finishing.
    if (a.rows == nullptr && a.route == nullptr && gwarp < n_chunks && lane < prefetch_rows) {
        const int p = gwarp * kChunk + lane;
        if (p < a.n_rows)
            prefetch_l2_bulk(static_cast<const T*>(a.ex[0].wg) + (size_t)p * d,
                             (unsigned)(d * sizeof(T)));
    }
    pdl_wait();
    pdl_launch_dependents();

    resolve_experts(a, es);
    const int n_x = a.route ? a.batch : a.nt;
    const int x_tok0 = a.route ? 0 : a.tok0;
    for (int t = 0; t < n_x; ++t) {
        if (a.norm_from_h) {
            block_rmsnorm<T>(a.h + (size_t)(x_tok0 + t) * d, d, xs + (size_t)t * d, red);
        } else {
            for (int i = threadIdx.x; i < d; i += blockDim.x)
                xs[(size_t)t * d + i] = Vec<T>::load1(a.x, (size_t)(x_tok0 + t) * d + i);
        }
    }
    __syncthreads();

    const int n_items = es.n_act * n_chunks;
    for (int item = gwarp; item < n_items; item += nwarps) {
        const int ea = item / n_chunks;
        const int chunk = item - ea * n_chunks;
        const int e = es.act[ea];
        const int ntok = es.ntok[e];
        const T* __restrict__ wg = static_cast<const T*>(a.ex[e].wg);
        const T* __restrict__ wu = static_cast<const T*>(a.ex[e].wu);
        int xo[NT];
#pragma unroll
        for (int k = 0; k < NT; ++k) {
            const int t = k < ntok ? (a.route ? es.tok[e][k] : k) : 0;
            xo[k] = t * d;
        }

        // lane r < kChunk: neuron id of row position p0 + r (-1: none)
        const int p0 = chunk * kChunk;
        int jr = -1;
        if (lane < kChunk && p0 + lane < a.n_rows) {
            const int p = p0 + lane;
            if (a.rows != nullptr) {
                const int j = a.rows[p];
                const bool ok = (unsigned)j < (unsigned)a.m && (p == 0 || a.rows[p - 1] < j);
                if (ok)
                    jr = j;
                else
                    atomicOr(a.status, kStatusBadIndex);
            } else {
                jr = p;
            }
        }

        // 1. gate pre-activations of the chunk's rows
        float greg[NT];
#pragma unroll
        for (int k = 0; k < NT; ++k) greg[k] = 0.0f;
#pragma unroll
        for (int g0 = 0; g0 < kChunk; g0 += R) {
            int row[R];
#pragma unroll
            for (int r = 0; r < R; ++r) row[r] = __shfl_sync(0xffffffffu, jr, g0 + r);
            float acc[R][NT];
            rows_dot<T, NT, R, U>(wg, row, d, xs, xo, ntok, lane, acc);
#pragma unroll
            for (int r = 0; r < R; ++r)
                if (lane == g0 + r)
#pragma unroll
                    for (int k = 0; k < NT; ++k) greg[k] = acc[r][k];
        }

        // 2. gate-active rows: any token with g > 0
        bool ga = false;
#pragma unroll
        for (int k = 0; k < NT; ++k) ga |= (k < ntok) && (greg[k] > 0.0f);
        ga = ga && jr >= 0;
        const unsigned gm = __ballot_sync(0xffffffffu, ga);

        // 3. up pre-activations, gathered over the gate-active rows only
        float ureg[NT];
#pragma unroll
        for (int k = 0; k < NT; ++k) ureg[k] = 0.0f;
        unsigned rest = gm;
        while (rest) {
            int row[R];
            int slot[R];
#pragma unroll
            for (int r = 0; r < R; ++r) {
                if (rest) {
                    const int b = __ffs(rest) - 1;
                    rest &= rest - 1u;
                    slot[r] = b;
                    row[r] = __shfl_sync(0xffffffffu, jr, b);
                } else {
                    slot[r] = -1;
                    row[r] = -1;
                }
            }
            float acc[R][NT];
            rows_dot<T, NT, R, U>(wu, row, d, xs, xo, ntok, lane, acc);
#pragma unroll
            for (int r = 0; r < R; ++r)
                if (lane == slot[r])
#pragma unroll
                    for (int k = 0; k < NT; ++k) ureg[k] = acc[r][k];
        }

        // 4. per-token masks, union byte, and c = w * g * u for union rows
        const bool mine = ga;  // lane's row is gate-active for some token
        unsigned ub = 0u;
        uint8_t* gb = a.gbits + (size_t)e * a.bits_expert_stride + chunk;
        uint8_t* bb = a.bbits + (size_t)e * a.bits_expert_stride + chunk;
#pragma unroll
        for (int k = 0; k < NT; ++k) {
            if (k < ntok) {
                const bool gk = jr >= 0 && greg[k] > 0.0f;
                const bool bk = mine && gk && ureg[k] > 0.0f;
                const unsigned gbyte = __ballot_sync(0xffffffffu, gk) & 0xffu;
                const unsigned bbyte = __ballot_sync(0xffffffffu, bk) & 0xffu;
                ub |= bbyte;
                if (lane == 0) {
                    const size_t tb = (size_t)(a.bits_tok_base + k) * a.nbytes;
                    gb[tb] = (uint8_t)gbyte;
                    bb[tb] = (uint8_t)bbyte;
                }
            }
        }
        if (lane == 0) {
            a.ubits[(size_t)e * a.nbytes + chunk] = (uint8_t)ub;
            a.ugbits[(size_t)e * a.nbytes + chunk] = (uint8_t)gm;
        }
        // c by batch slot: the pass-local token (single FFN) or the global
        // token (MoE, 0 for tokens not routed to this expert)
        if (lane < kChunk && ((ub >> lane) & 1u)) {
            float* cv = a.cval + ((size_t)e * kMaxPass) * a.cval_tok_stride + p0 + lane;
            float val[NT];
#pragma unroll
            for (int k = 0; k < NT; ++k)
                val[k] = (k < ntok && greg[k] > 0.0f && ureg[k] > 0.0f) ? es.w[e][k] * (greg[k] * ureg[k])
                                                                         : 0.0f;
            if (a.route == nullptr) {
#pragma unroll
                for (int k = 0; k < NT; ++k)
                    if (k < ntok) cv[(size_t)k * a.cval_tok_stride] = val[k];
            } else {
                for (int t = 0; t < a.batch; ++t) {
                    float v = 0.0f;
#pragma unroll
                    for (int k = 0; k < NT; ++k)
                        if (k < ntok && es.tok[e][k] == t) v = val[k];
                    cv[(size_t)t * a.cval_tok_stride] = v;
                }
            }
        }
    }
}

template <typename T, int NT>
static cudaError_t launch_t(const FfnLaunch& a, int grid, cudaStream_t stream, bool pdl) {
    const int n_x = a.route ? a.batch : a.nt;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kGateUpWarps * kWarp);
    cfg.dynamicSmemBytes = (size_t)n_x * a.d * sizeof(float);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    const int prefetch_rows = 2;
    return cudaLaunchKernelEx(&cfg, k_gate_up<T, NT>, a, prefetch_rows);
}

// Allow the largest dynamic shared memory the device offers (minus the
// kernel's static shared memory) for every instantiation.
template <typename T, int NT>
static cudaError_t prepare_t(int optin) {
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, k_gate_up<T, NT>);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(k_gate_up<T, NT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                optin - (int)fa.sharedSizeBytes);
}

cudaError_t prepare_gate_up(int optin_smem) {
    cudaError_t e = cudaSuccess;
    if (e == cudaSuccess) e = prepare_t<__nv_bfloat16, 1>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<__nv_bfloat16, 2>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<__nv_bfloat16, 4>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<__nv_bfloat16, 8>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<float, 1>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<float, 2>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<float, 4>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<float, 8>(optin_smem);
    return e;
}

cudaError_t launch_gate_up(const FfnLaunch& a, int wdtype, int pass_tokens, int grid,
                           cudaStream_t stream, bool pdl) {
    if (wdtype == 1) {
        switch (pass_tokens) {
            case 1: return launch_t<__nv_bfloat16, 1>(a, grid, stream, pdl);
            case 2: return launch_t<__nv_bfloat16, 2>(a, grid, stream, pdl);
            case 4: return launch_t<__nv_bfloat16, 4>(a, grid, stream, pdl);
            case 8: return launch_t<__nv_bfloat16, 8>(a, grid, stream, pdl);
        }
    } else {
        switch (pass_tokens) {
            case 1: return launch_t<float, 1>(a, grid, stream, pdl);
            case 2: return launch_t<float, 2>(a, grid, stream, pdl);
            case 4: return launch_t<float, 4>(a, grid, stream, pdl);
            case 8: return launch_t<float, 8>(a, grid, stream, pdl);
        }
    }
    return cudaErrorInvalidValue;
}

template <typename T, int NT>
static int occupancy_t(size_t smem) {
    int nb = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, k_gate_up<T, NT>, kGateUpWarps * kWarp,
                                                      smem) != cudaSuccess)
        return 1;
    return nb > 0 ? nb : 1;
}

int gate_up_blocks_per_sm(int wdtype, int pass_tokens, int x_tokens, int d) {
    const size_t smem = (size_t)x_tokens * d * sizeof(float);
    if (wdtype == 1) {
        switch (pass_tokens) {
            case 1: return occupancy_t<__nv_bfloat16, 1>(smem);
            case 2: return occupancy_t<__nv_bfloat16, 2>(smem);
            case 4: return occupancy_t<__nv_bfloat16, 4>(smem);
            default: return occupancy_t<__nv_bfloat16, 8>(smem);
        }
    }
    switch (pass_tokens) {
        case 1: return occupancy_t<float, 1>(smem);
        case 2: return occupancy_t<float, 2>(smem);
        case 4: return occupancy_t<float, 4>(smem);
        default: return occupancy_t<float, 8>(smem);
    }
}

}  // namespace tsffn
