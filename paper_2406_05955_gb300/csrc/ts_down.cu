// ts_down.cu -- gathered down projection y = sum_{j active} c_j W_down[j,:]
// (the "Combined(x) W_down" of Eq. 1, restricted to the non-zero dReLU
// activations of Eq. 2).
//
// Grid (n_cs, n_rg): blockIdx.x picks a slice of kColSlice output columns,
// blockIdx.y one of n_rg equal shares of the ordered active list. The list is
// not materialised in global memory: every CTA reads the union bitmap words
// (expert-major, row order), prefix-sums their popcounts and pulls out the
// entries of its share. Each warp takes every kDownWarps-th entry and reads
// that row's 512-byte (bf16) or 1 KB (fp32) column segment with 16-byte
// loads, accumulating c * w in fp32 registers per token. The CTA sums its
// warps in shared memory, writes one partial per (share, token, column), and
// the last CTA of the column slice to finish (atomic ticket) adds the n_rg
// partials in share order -- a fixed order, so y is bitwise reproducible.
#include "ts_kernels.cuh"

namespace tsffn {

constexpr int kListCap = 1024;  // entries a CTA stages in shared memory at once
constexpr int kDownUnroll = 4;  // rows a warp has in flight

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
    constexpr int V = kColSlice / (kWarp * VEC);  // 16-byte loads per lane per row
    constexpr int VPL = V * VEC;                  // columns per lane
    extern __shared__ __align__(16) float red[];  // [kDownWarps][NT][kColSlice]
    __shared__ ExpertSets es;
    __shared__ int2 s_list[kListCap];
    __shared__ int s_scan[kDownWarps];
    __shared__ int s_total;
    __shared__ int s_last;

    pdl_wait();
    pdl_launch_dependents();
    resolve_experts(a, es);

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int tid = threadIdx.x;
    const int nthr = blockDim.x;
    const int d = a.d;
    const int cs = blockIdx.x;
    const int rg = blockIdx.y;
    const int n_rg = gridDim.y;
    const int nwords = (a.n_rows + 31) / 32;
    const int total_words = es.n_act * nwords;

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
    const int r0 = (int)((long long)N * rg / n_rg);
    const int r1 = (int)((long long)N * (rg + 1) / n_rg);

    // local token slot of each (expert, token): route ? global token : pass-local index
    float acc[NT][VPL];
#pragma unroll
    for (int k = 0; k < NT; ++k)
#pragma unroll
        for (int c = 0; c < VPL; ++c) acc[k][c] = 0.0f;

    const int col_base = cs * kColSlice;
    for (int s = r0; s < r1; s += kListCap) {
        const int s1 = min(s + kListCap, r1);
        if (cnt > 0 && off < s1 && off + cnt > s) {
            int rank = off;
            for (int w = w0; w < w1 && rank < s1; ++w) {
                unsigned bits = union_word(a, es, nwords, w);
                while (bits && rank < s1) {
                    const int b = __ffs(bits) - 1;
                    bits &= bits - 1u;
                    if (rank >= s) {
                        const int ea = w / nwords;
                        const int pos = (w - ea * nwords) * 32 + b;
                        s_list[rank - s] = make_int2(ea, pos);
                    }
                    ++rank;
                }
            }
        }
        __syncthreads();
        const int n = s1 - s;
        for (int i0 = warp; i0 < n; i0 += kDownWarps * kDownUnroll) {
            uint4 wv[kDownUnroll][V];
            int ent_e[kDownUnroll], ent_p[kDownUnroll];
#pragma unroll
            for (int q = 0; q < kDownUnroll; ++q) {
                const int i = i0 + q * kDownWarps;
                ent_e[q] = -1;
                ent_p[q] = 0;
                if (i < n) {
                    const int2 en = s_list[i];
                    const int e = es.act[en.x];
                    ent_e[q] = e;
                    ent_p[q] = en.y;
                    const int j = a.rows ? a.rows[en.y] : en.y;
                    const T* row = static_cast<const T*>(a.ex[e].wd) + (size_t)j * d;
#pragma unroll
                    for (int v = 0; v < V; ++v) {
                        const int col = col_base + v * kWarp * VEC + lane * VEC;
                        wv[q][v] = col < d ? ld_stream(row + col) : make_uint4(0u, 0u, 0u, 0u);
                    }
                } else {
#pragma unroll
                    for (int v = 0; v < V; ++v) wv[q][v] = make_uint4(0u, 0u, 0u, 0u);
                }
            }
#pragma unroll
            for (int q = 0; q < kDownUnroll; ++q) {
                const int e = ent_e[q];
                if (e < 0) continue;
                const int ntok = es.ntok[e];
                const float* cv = a.cval + ((size_t)e * kMaxPass) * a.cval_tok_stride + ent_p[q];
                float f[V][VEC];
#pragma unroll
                for (int v = 0; v < V; ++v) Vec<T>::unpack(wv[q][v], f[v]);
#pragma unroll
                for (int k = 0; k < NT; ++k) {
                    if (k < ntok) {
                        const float c = cv[(size_t)k * a.cval_tok_stride];
                        const int slot = a.route ? es.tok[e][k] : k;
                        // slot < NT always: MoE batches are <= NT tokens, passes are NT wide
#pragma unroll
                        for (int s2 = 0; s2 < NT; ++s2) {
                            if (s2 == slot) {
#pragma unroll
                                for (int v = 0; v < V; ++v)
#pragma unroll
                                    for (int c2 = 0; c2 < VEC; ++c2)
                                        acc[s2][v * VEC + c2] = fmaf(c, f[v][c2], acc[s2][v * VEC + c2]);
                            }
                        }
                    }
                }
            }
        }
        __syncthreads();
    }

    // block reduction over warps (fixed order) -> partial of this share
    const int n_slots = a.route ? a.batch : a.nt;
#pragma unroll
    for (int k = 0; k < NT; ++k)
#pragma unroll
        for (int v = 0; v < V; ++v)
#pragma unroll
            for (int c2 = 0; c2 < VEC; ++c2)
                red[((size_t)warp * NT + k) * kColSlice + v * kWarp * VEC + lane * VEC + c2] =
                    acc[k][v * VEC + c2];
    __syncthreads();
    for (int idx = tid; idx < n_slots * kColSlice; idx += nthr) {
        const int k = idx / kColSlice;
        const int c = idx - k * kColSlice;
        const int col = col_base + c;
        if (col >= d) continue;
        float sum = 0.0f;
        for (int w = 0; w < kDownWarps; ++w) sum += red[((size_t)w * NT + k) * kColSlice + c];
        a.partial[((size_t)rg * kMaxPass + k) * d + col] = sum;
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) {
        const unsigned prev = atomicAdd(&a.counters[cs], 1u);
        s_last = (prev == (unsigned)(n_rg - 1));
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    for (int idx = tid; idx < n_slots * kColSlice; idx += nthr) {
        const int k = idx / kColSlice;
        const int c = idx - k * kColSlice;
        const int col = col_base + c;
        if (col >= d) continue;
        float sum = 0.0f;
        for (int r = 0; r < n_rg; ++r) sum += __ldcg(&a.partial[((size_t)r * kMaxPass + k) * d + col]);
        const int tok = a.route ? k : a.tok0 + k;
        if (a.residual_out)
            a.h[(size_t)tok * d + col] += sum;
        else
            a.y[(size_t)tok * d + col] = sum;
    }
    if (tid == 0) a.counters[cs] = 0u;  // ticket ready for the next launch
}

template <typename T, int NT>
static cudaError_t launch_t(const FfnLaunch& a, cudaStream_t stream, bool pdl) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.n_cs, a.n_rg);
    cfg.blockDim = dim3(kDownWarps * kWarp);
    cfg.dynamicSmemBytes = (size_t)kDownWarps * NT * kColSlice * sizeof(float);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, k_down<T, NT>, a);
}

template <typename T, int NT>
static cudaError_t prepare_t() {
    return cudaFuncSetAttribute(k_down<T, NT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)(kDownWarps * NT * kColSlice * sizeof(float)));
}

cudaError_t prepare_down() {
    cudaError_t e = cudaSuccess;
    if (e == cudaSuccess) e = prepare_t<__nv_bfloat16, 1>();
    if (e == cudaSuccess) e = prepare_t<__nv_bfloat16, 2>();
    if (e == cudaSuccess) e = prepare_t<__nv_bfloat16, 4>();
    if (e == cudaSuccess) e = prepare_t<__nv_bfloat16, 8>();
    if (e == cudaSuccess) e = prepare_t<float, 1>();
    if (e == cudaSuccess) e = prepare_t<float, 2>();
    if (e == cudaSuccess) e = prepare_t<float, 4>();
    if (e == cudaSuccess) e = prepare_t<float, 8>();
    return e;
}

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
