// ts_down.cu -- gathered down projection y = sum_{j active} c_j W_down[j,:]
// (the "Combined(x) W_down" of Eq. 1, restricted to the non-zero dReLU
// activations of Eq. 2).
//
// Passes of up to kAccMaxTokens tokens: the gate+up CTAs have already summed
// their own rows; k_down_reduce (below) adds their partials. Wider passes:
// k_down gathers the rows itself. One CTA per slice of kDownCols output columns: 64 bytes of every active
// row (32 bf16 or 16 fp32 columns). Every CTA reads the union bitmap words
// (expert-major, row order), prefix-sums their popcounts and stages the
// ordered (expert, row) entries in shared memory. A warp instruction covers
// 8 entries (4 lanes x 16 bytes per row segment); each of the 16 warps keeps
// up to 12 such instructions in flight (the whole list at batch 1 and ~10%
// activation, in one round trip; the gate+up kernel has already pulled the
// rows into L2), accumulating c * w in fp32 registers per
// batch slot. Rows are reduced across lanes (shuffles) and warps (shared
// memory) in a fixed order and written straight to y (or added to the
// residual): no partial buffers, no cross-CTA hand-off, bitwise reproducible.
#include "ts_kernels.cuh"

namespace tsffn {

constexpr int kListCap = 2048;  // entries a CTA stages in shared memory at once
constexpr int kLanesPerRow = 4;
constexpr int kRowsPerInst = kWarp / kLanesPerRow;  // 8

template <int NT>
struct DownShape {
    static constexpr int U = NT <= 2 ? 12 : (NT == 4 ? 8 : 4);  // row groups in flight per warp
};

__device__ __forceinline__ unsigned union_word(const FfnLaunch& a, const ExpertSets& es,
                                               int nwords, int w) {
    const int ea = w / nwords;
    const int wi = w - ea * nwords;
    const int e = es.act[ea];
    unsigned bits = *reinterpret_cast<const unsigned*>(a.ubits + (size_t)e * a.nbytes + (size_t)wi * 4);
    const int left = a.n_rows - wi * 32;  // rows of the row space in this word
    if (left < 32) bits &= (1u << left) - 1u;
    return bits;
}

template <typename T, int NT>
__global__ void __launch_bounds__(kDownWarps * kWarp) k_down(const FfnLaunch a) {
    constexpr int VEC = Vec<T>::N;
    constexpr int COLS = kLanesPerRow * VEC;  // columns per CTA (64 bytes of a row)
    constexpr int U = DownShape<NT>::U;
    __shared__ ExpertSets es;
    __shared__ int2 s_list[kListCap];
    __shared__ int s_scan[kDownWarps];
    __shared__ int s_total;
    __shared__ float red[kDownWarps][NT][COLS];

    if (a.next_wg != nullptr && a.prefetch_rows > 0) {
        // independent of the previous kernel: the next layer's weights
        const int nc = (a.next_n_rows + kChunk - 1) / kChunk;
        const unsigned row_bytes = (unsigned)(a.d * sizeof(T));
        const T* nw = static_cast<const T*>(a.next_wg);
        for (int b = blockIdx.x; b < a.next_grid; b += gridDim.x) {
            const int r0 = (int)((long long)nc * b / a.next_grid) * kChunk;
            const int r1 = min((int)((long long)nc * (b + 1) / a.next_grid) * kChunk, a.next_n_rows);
            const int rn = min(r1 - r0, a.prefetch_rows);
            const int r = (int)threadIdx.x * kChunk;
            if (r < rn)
                prefetch_l2_bulk(nw + (size_t)(r0 + r) * a.d, (unsigned)min(kChunk, rn - r) * row_bytes);
        }
    }
    pdl_wait();
    pdl_launch_dependents();
    resolve_experts(a, es);

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int tid = threadIdx.x;
    const int nthr = blockDim.x;
    const int d = a.d;
    const int nwords = (a.n_rows + 31) / 32;
    const int total_words = es.n_act * nwords;
    const int n_slots = a.route ? a.batch : a.nt;

    // contiguous word range per thread, popcount, block exclusive scan
    const int per = (total_words + nthr - 1) / nthr;
    const int w0 = min(tid * per, total_words);
    const int w1 = min(w0 + per, total_words);
    int cnt = 0;
    for (int w = w0; w < w1; ++w) cnt += __popc(union_word(a, es, nwords, w));
    int incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
    }
    if (lane == 31) s_scan[warp] = incl;
    __syncthreads();
    if (tid == 0) {
        int run = 0;
        for (int w = 0; w < kDownWarps; ++w) {
            const int v = s_scan[w];
            s_scan[w] = run;
            run += v;
        }
        s_total = run;
    }
    __syncthreads();
    const int off = s_scan[warp] + incl - cnt;  // rank of this thread's first entry
    const int N = s_total;

    const int col = blockIdx.x * COLS + (lane & (kLanesPerRow - 1)) * VEC;
    const int slot_in_inst = lane / kLanesPerRow;
    float acc[NT][VEC];
#pragma unroll
    for (int k = 0; k < NT; ++k)
#pragma unroll
        for (int c = 0; c < VEC; ++c) acc[k][c] = 0.0f;

    for (int s = 0; s < N; s += kListCap) {
        const int s1 = min(s + kListCap, N);
        if (cnt > 0 && off < s1 && off + cnt > s) {
            int rank = off;
            for (int w = w0; w < w1 && rank < s1; ++w) {
                unsigned bits = union_word(a, es, nwords, w);
                while (bits && rank < s1) {
                    const int b = __ffs(bits) - 1;
                    bits &= bits - 1u;
                    if (rank >= s) {
                        const int ea = w / nwords;
                        s_list[rank - s] = make_int2(ea, (w - ea * nwords) * 32 + b);
                    }
                    ++rank;
                }
            }
        }
        __syncthreads();
        const int n = s1 - s;
        const int n_inst = (n + kRowsPerInst - 1) / kRowsPerInst;
        for (int g0 = warp; g0 < n_inst; g0 += kDownWarps * U) {
            uint4 wv[U];
            float cv[U][NT];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int i = (g0 + u * kDownWarps) * kRowsPerInst + slot_in_inst;
                wv[u] = make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
                for (int k = 0; k < NT; ++k) cv[u][k] = 0.0f;
                if (i < n) {
                    const int2 en = s_list[i];
                    const int e = es.act[en.x];
                    const int j = debug_row(a.rows ? a.rows[en.y] : en.y, a.m, a.status);
                    if (col < d)
                        wv[u] = ld_stream(static_cast<const T*>(a.ex[e].wd) + (size_t)j * d + col);
                    const float* cp = a.cval + ((size_t)e * kMaxPass) * a.cval_tok_stride + en.y;
#pragma unroll
                    for (int k = 0; k < NT; ++k)
                        if (k < n_slots) cv[u][k] = cp[(size_t)k * a.cval_tok_stride];
                }
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                float f[VEC];
                Vec<T>::unpack(wv[u], f);
#pragma unroll
                for (int k = 0; k < NT; ++k)
#pragma unroll
                    for (int c = 0; c < VEC; ++c) acc[k][c] = fmaf(cv[u][k], f[c], acc[k][c]);
            }
        }
        __syncthreads();
    }

    // reduce over the 8 row slots of a warp (lanes with equal lane % 4), then over warps
#pragma unroll
    for (int k = 0; k < NT; ++k)
#pragma unroll
        for (int c = 0; c < VEC; ++c) {
            float v = acc[k][c];
            v += __shfl_xor_sync(0xffffffffu, v, 4);
            v += __shfl_xor_sync(0xffffffffu, v, 8);
            v += __shfl_xor_sync(0xffffffffu, v, 16);
            acc[k][c] = v;
        }
    if (lane < kLanesPerRow) {
#pragma unroll
        for (int k = 0; k < NT; ++k)
#pragma unroll
            for (int c = 0; c < VEC; ++c) red[warp][k][lane * VEC + c] = acc[k][c];
    }
    __syncthreads();
    for (int idx = tid; idx < n_slots * COLS; idx += nthr) {
        const int k = idx / COLS;
        const int c = idx - k * COLS;
        const int cc = blockIdx.x * COLS + c;
        if (cc >= d) continue;
        float sum = 0.0f;
#pragma unroll
        for (int w = 0; w < kDownWarps; ++w) sum += red[w][k][c];
        const int tok = a.route ? k : a.tok0 + k;
        if (a.residual_out)
            a.h[(size_t)tok * d + cc] += sum;
        else
            a.y[(size_t)tok * d + cc] = sum;
    }
}

template <typename T, int NT>
static cudaError_t launch_t(const FfnLaunch& a, cudaStream_t stream, bool pdl) {
    constexpr int COLS = kLanesPerRow * Vec<T>::N;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((a.d + COLS - 1) / COLS);
    cfg.blockDim = dim3(kDownWarps * kWarp);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, k_down<T, NT>, a);
}

// ---------------------------------------------------------------------------
// Passes of <= kAccMaxTokens tokens: every gate+up CTA has already summed
// c_j W_down[j,:] over its own both-active rows (its accumulator warp) into
// its block of the partial buffer. Here the blocks are added in CTA order:
// one CTA per 64 output columns, a half-warp covers them with 16-byte loads,
// the 32 half-warps take every 32nd block, and the half-warp and warp sums
// are combined in a fixed order (bitwise reproducible).
// ---------------------------------------------------------------------------
constexpr int kRedCols = 64;
constexpr int kRedThreads = 512;
constexpr int kRedWarps = kRedThreads / kWarp;
constexpr int kRedLanes = kRedCols / 4;  // lanes of a half-warp, a float4 each
constexpr int kRedBatch = 6;  // partial blocks a half-warp has in flight

template <int NT>
__global__ void __launch_bounds__(kRedThreads) k_down_reduce(const FfnLaunch a) {
    __shared__ float4 red[kRedWarps][NT][kRedLanes];
    // In an FFN stack the next kernel is the next layer's gate+up kernel: it
    // may be scheduled at once (it waits for this one to finish before it
    // reads h), and its CTAs take each SM as the gate+up CTA there exits, so
    // its prologue (launch, list set-up) overlaps this reduction.
    if (a.trigger_early) pdl_launch_dependents();
    pdl_wait();
    if (!a.trigger_early) pdl_launch_dependents();
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int hw = lane / kRedLanes;
    const int cl = lane % kRedLanes;
    const int d = a.d;
    const int n_slots = a.route ? a.batch : a.nt;
    const int col = blockIdx.x * kRedCols + cl * 4;
    const bool valid = col < d;

    // this thread's output (n_slots * kRedCols <= kRedThreads): its residual
    // is read while the partials load
    const int out_k = threadIdx.x / kRedCols;
    const int out_c = blockIdx.x * kRedCols + (threadIdx.x - out_k * kRedCols);
    const bool has_out = out_k < n_slots && out_c < d;
    const size_t out_i = (size_t)(a.route ? out_k : a.tok0 + out_k) * d + out_c;
    float h_old = 0.0f;
    if (has_out && a.residual_out) h_old = a.h[out_i];

    float4 acc[NT];
#pragma unroll
    for (int k = 0; k < NT; ++k) acc[k] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    if (valid) {
        // this half-warp's partial blocks b = warp * 2 + hw + i * 2 * kRedWarps:
        // kRedBatch of them loaded at once, then added in the same order
        const size_t cta_stride = (size_t)a.partial_slots * d;
        constexpr int kStride = 2 * kRedWarps;
        for (int b0 = warp * 2 + hw; b0 < a.partial_ctas; b0 += kRedBatch * kStride) {
            float4 v[kRedBatch][NT];
#pragma unroll
            for (int i = 0; i < kRedBatch; ++i) {
                const int b = b0 + i * kStride;
                const float* p = a.partial + (size_t)b * cta_stride + col;
#pragma unroll
                for (int k = 0; k < NT; ++k)
                    v[i][k] = (b < a.partial_ctas && k < n_slots) ? *reinterpret_cast<const float4*>(p + (size_t)k * d)
                                                                  : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            }
#pragma unroll
            for (int i = 0; i < kRedBatch; ++i)
                if (b0 + i * kStride < a.partial_ctas) {
#pragma unroll
                    for (int k = 0; k < NT; ++k)
                        if (k < n_slots) {
                            acc[k].x += v[i][k].x;
                            acc[k].y += v[i][k].y;
                            acc[k].z += v[i][k].z;
                            acc[k].w += v[i][k].w;
                        }
                }
        }
    }
#pragma unroll
    for (int k = 0; k < NT; ++k) {
        // half-warp 0 + half-warp 1: both halves end with the same sum
        acc[k].x += __shfl_xor_sync(0xffffffffu, acc[k].x, kRedLanes);
        acc[k].y += __shfl_xor_sync(0xffffffffu, acc[k].y, kRedLanes);
        acc[k].z += __shfl_xor_sync(0xffffffffu, acc[k].z, kRedLanes);
        acc[k].w += __shfl_xor_sync(0xffffffffu, acc[k].w, kRedLanes);
    }
    if (hw == 0) {
#pragma unroll
        for (int k = 0; k < NT; ++k) red[warp][k][cl] = acc[k];
    }
    __syncthreads();
    if (has_out) {
        const int c = out_c - blockIdx.x * kRedCols;
        float sum = 0.0f;
#pragma unroll
        for (int w = 0; w < kRedWarps; ++w) sum += reinterpret_cast<const float*>(&red[w][out_k][0])[c];
        if (a.residual_out)
            a.h[out_i] = h_old + sum;
        else
            a.y[out_i] = sum;
    }
}

template <int NT>
static cudaError_t launch_reduce_t(const FfnLaunch& a, cudaStream_t stream, bool pdl) {
    static_assert(NT * kRedCols <= kRedThreads, "one output per thread");
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((a.d + kRedCols - 1) / kRedCols);
    cfg.blockDim = dim3(kRedThreads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, k_down_reduce<NT>, a);
}

cudaError_t launch_down_reduce(const FfnLaunch& a, int pass_tokens, cudaStream_t stream, bool pdl) {
    if (a.partial == nullptr || a.partial_ctas < 1) return cudaErrorInvalidValue;
    switch (pass_tokens) {
        case 1: return launch_reduce_t<1>(a, stream, pdl);
        case 2: return launch_reduce_t<2>(a, stream, pdl);
    }
    return cudaErrorInvalidValue;
}

cudaError_t prepare_down() { return cudaSuccess; }

cudaError_t launch_down(const FfnLaunch& a, int wdtype, int pass_tokens, cudaStream_t stream,
                        bool pdl) {
    if (wdtype == 1) {
        switch (pass_tokens) {
            case 1: return launch_t<__nv_bfloat16, 1>(a, stream, pdl);
            case 2: return launch_t<__nv_bfloat16, 2>(a, stream, pdl);
            case 4: return launch_t<__nv_bfloat16, 4>(a, stream, pdl);
            case 8: return launch_t<__nv_bfloat16, 8>(a, stream, pdl);
        }
    } else {
        switch (pass_tokens) {
            case 1: return launch_t<float, 1>(a, stream, pdl);
            case 2: return launch_t<float, 2>(a, stream, pdl);
            case 4: return launch_t<float, 4>(a, stream, pdl);
            case 8: return launch_t<float, 8>(a, stream, pdl);
        }
    }
    return cudaErrorInvalidValue;
}

}  // namespace tsffn
