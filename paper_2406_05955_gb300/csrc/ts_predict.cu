// ts_predict.cu -- the activation predictor of Sec. 7 on the device.
//
// A predictor is a two-layer ReLU MLP over the FFN's input x:
//     hid = max(0, W1 x)          W1 [r][d]
//     s   = W2 hid                W2 [m][r]   (one score per neuron)
// For a batch, a neuron's key is its largest score over the tokens; the K
// neurons with the largest keys (a lower neuron index winning a tie) form the
// list, written in ascending neuron order, that the FFN kernels' predictor mode
// consumes. Three launches chained with programmatic dependent launch:
//   k_pred_hidden  W1 GEMV per K-segment into fp32 partials (HBM-bound: reads W1 once)
//   k_pred_score   partial sum + ReLU, W2 GEMV, max over tokens, order-preserving
//                  key bits (HBM-bound: reads W2 once)
//   k_pred_select  one CTA: MSB-first 8-bit radix select of the K-th largest
//                  key, then an ordered emission of the selected ids
//                  (k_pred_select_hist, led by the score kernel's histogram,
//                  when m <= 16384)
#include <math.h>

#include <algorithm>

#include "ts_kernels.cuh"
#include "ts_predict.h"

namespace tsffn {
namespace {

constexpr int kPredThreads = 256;
constexpr int kPredWarps = kPredThreads / kWarp;
constexpr int kSelThreads = 1024;
constexpr int kSelWarps = kSelThreads / kWarp;
// keys staged in shared memory by the select kernel when m * 4 bytes fit
constexpr int kSelSmemMax = 200 * 1024;
constexpr int kSmemSlack = 1024;
// the select kernel's shared-memory cap on this device (set by prepare_predict)
int g_sel_smem = 0;

int pow2_batch(int b) { return b <= 1 ? 1 : b <= 2 ? 2 : b <= 4 ? 4 : 8; }

// `n` fp32 activations at `xr` times the unpacked weights `w`, into acc.
template <int N>
__device__ __forceinline__ float dot_vec(const float (&w)[N], const float* __restrict__ xr, float acc) {
#pragma unroll
    for (int e = 0; e < N; e += 4) {
        const float4 q = *reinterpret_cast<const float4*>(xr + e);
        acc = fmaf(w[e], q.x, acc);
        acc = fmaf(w[e + 1], q.y, acc);
        acc = fmaf(w[e + 2], q.z, acc);
        acc = fmaf(w[e + 3], q.w, acc);
    }
    return acc;
}

// Hidden layer: warp-sized pieces (row of W1, K-segment); each lane streams
// 16-byte vectors of the row, up to 8 in flight, against the x rows held in
// shared memory as fp32 (tokens batch .. NB-1 are zero).
template <typename T, int NB>
__global__ void __launch_bounds__(kPredThreads) k_pred_hidden(const PredictLaunch p) {
    extern __shared__ __align__(16) float xs[];  // [NB][d]
    __shared__ float red[kPredWarps];
    constexpr int N = Vec<T>::N;
    const int d = p.d;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int steps = d / (kWarp * N) / p.splits;  // 16-byte vectors per lane per piece
    const int seg = steps * kWarp * N;
    const int total = p.r * p.splits;
    auto wrow_of = [&](int piece) {
        const int sp = piece / p.r, row = piece - sp * p.r;
        return static_cast<const T*>(p.w1) + (size_t)row * d + (size_t)sp * seg + lane * N;
    };
    // W1 does not depend on earlier kernels: the first vectors of this warp's
    // first piece are loaded before the wait, while the previous kernel ends.
    int piece = blockIdx.x * kPredWarps + warp;
    uint4 v[8];
    if (piece < total) {
        const T* wrow = wrow_of(piece);
#pragma unroll
        for (int u = 0; u < 8; ++u)
            v[u] = u < steps ? ld_stream(wrow + (size_t)u * kWarp * N) : make_uint4(0u, 0u, 0u, 0u);
    }
    pdl_launch_dependents();
    pdl_wait();
    // the select of the previous prediction has finished with the histogram
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < kPredHistParts * kPredHistBins;
         i += gridDim.x * blockDim.x)
        p.hist[i] = 0u;
    if (p.h != nullptr) {
        for (int t = 0; t < NB; ++t) {
            if (t < p.batch) {
                block_rmsnorm<T>(p.h + (size_t)t * d, d, xs + (size_t)t * d, red);
            } else {
                for (int i = threadIdx.x; i < d; i += blockDim.x) xs[(size_t)t * d + i] = 0.0f;
            }
        }
    } else {
        for (int i = threadIdx.x; i < NB * d; i += blockDim.x)
            xs[i] = i < p.batch * d ? Vec<T>::load1(p.x, (size_t)i) : 0.0f;
    }
    __syncthreads();

    bool loaded = true;  // v holds the first vectors of this piece
    for (; piece < total; piece += gridDim.x * kPredWarps) {
        const int sp = piece / p.r, row = piece - sp * p.r;
        const T* wrow = wrow_of(piece);
        const float* xb = xs + (size_t)sp * seg + lane * N;
        float acc[NB];
#pragma unroll
        for (int t = 0; t < NB; ++t) acc[t] = 0.0f;
        for (int s0 = 0; s0 < steps; s0 += 8) {
            if (!loaded) {
#pragma unroll
                for (int u = 0; u < 8; ++u)
                    v[u] = s0 + u < steps ? ld_stream(wrow + (size_t)(s0 + u) * kWarp * N)
                                          : make_uint4(0u, 0u, 0u, 0u);
            }
            loaded = false;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                if (s0 + u < steps) {
                    float w[N];
                    Vec<T>::unpack(v[u], w);
#pragma unroll
                    for (int t = 0; t < NB; ++t)
                        acc[t] = dot_vec<N>(w, xb + (size_t)t * d + (s0 + u) * kWarp * N, acc[t]);
                }
            }
        }
#pragma unroll
        for (int t = 0; t < NB; ++t) acc[t] = warp_sum(acc[t]);
        if (lane == 0)
#pragma unroll
            for (int t = 0; t < NB; ++t)
                if (t < p.batch) p.hid[((size_t)sp * p.batch + t) * p.r + row] = acc[t];
    }
}

// fp32 -> unsigned with the same order (-0 folded into +0 first).
__device__ __forceinline__ unsigned order_key(float f) {
    const unsigned u = __float_as_uint(__fadd_rn(f, 0.0f));
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Scores: every CTA rebuilds hid = max(0, sum of the partials) in shared
// memory, then each warp takes groups of RG consecutive W2 rows (one
// contiguous run of RG * r weights, STEPS 16-byte vectors per lane per row).
template <typename T, int NB, int STEPS>
__global__ void __launch_bounds__(kPredThreads) k_pred_score(const PredictLaunch p) {
    extern __shared__ __align__(16) float hs[];  // [NB][r]
    constexpr int N = Vec<T>::N;
    constexpr int RG = STEPS >= 8 ? 1 : 8 / STEPS;
    constexpr int WARPS = kPredWarps;
    const int r = p.r, m = p.m;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int groups = (m + RG - 1) / RG;
    uint4 v[RG][STEPS];
    auto load = [&](int g) {
        const int j0 = g * RG;
#pragma unroll
        for (int q = 0; q < RG; ++q)
#pragma unroll
            for (int s = 0; s < STEPS; ++s)
                v[q][s] = j0 + q < m ? ld_stream(static_cast<const T*>(p.w2) + (size_t)(j0 + q) * r +
                                                 s * kWarp * N + lane * N)
                                     : make_uint4(0u, 0u, 0u, 0u);
    };
    // W2 does not depend on earlier kernels: this warp's first group of rows
    // is loaded before the wait, while the hidden-layer kernel runs.
    int g = blockIdx.x * WARPS + warp;
    if (g < groups) load(g);
    pdl_launch_dependents();
    pdl_wait();
    for (int i = threadIdx.x; i < NB * r; i += blockDim.x) {
        const int t = i / r, j = i - t * r;
        float s = 0.0f;
        if (t < p.batch) {
            for (int sp = 0; sp < p.splits; ++sp) s += p.hid[((size_t)sp * p.batch + t) * r + j];
            s = fmaxf(s, 0.0f);
        }
        hs[i] = s;
    }
    __syncthreads();

    bool loaded = true;
    for (; g < groups; g += gridDim.x * WARPS) {
        const int j0 = g * RG;
        if (!loaded) load(g);
        loaded = false;
        float acc[RG][NB];
#pragma unroll
        for (int q = 0; q < RG; ++q)
#pragma unroll
            for (int t = 0; t < NB; ++t) acc[q][t] = 0.0f;
#pragma unroll
        for (int q = 0; q < RG; ++q)
#pragma unroll
            for (int s = 0; s < STEPS; ++s) {
                float w[N];
                Vec<T>::unpack(v[q][s], w);
#pragma unroll
                for (int t = 0; t < NB; ++t)
                    acc[q][t] = dot_vec<N>(w, hs + (size_t)t * r + s * kWarp * N + lane * N, acc[q][t]);
            }
#pragma unroll
        for (int q = 0; q < RG; ++q) {
            const int j = j0 + q;
            float best = -INFINITY;
#pragma unroll
            for (int t = 0; t < NB; ++t) {
                const float sv = warp_sum(acc[q][t]);
                if (t < p.batch) {
                    best = fmaxf(best, sv);
                    if (p.scores != nullptr && lane == 0 && j < m) p.scores[(size_t)t * m + j] = sv;
                }
            }
            if (lane == 0 && j < m) {
                const unsigned k = order_key(best);
                p.key[j] = k;
                atomicAdd(&p.hist[(blockIdx.x % kPredHistParts) * kPredHistBins + (k >> 20)], 1u);
            }
        }
    }
}

// The K-th largest key T by an MSB-first radix select over 8-bit digits
// (a warp adds its lanes' equal digits with one shared-memory atomic), then
// the ids with key > T and the first (K - #{key > T}) ids with key == T, in
// ascending order: warps own contiguous id ranges, a scan over the warps gives
// each range's output offset, and ballots order the ids inside a range.
__global__ void __launch_bounds__(kSelThreads) k_pred_select(const PredictLaunch p, int staged) {
    extern __shared__ unsigned ks[];  // [m] when staged
    __shared__ unsigned hist[256];
    __shared__ unsigned wsum[8];
    __shared__ unsigned s_prefix, s_mask;
    __shared__ int s_rem;
    __shared__ int s_gt[kSelWarps], s_eq[kSelWarps];
    pdl_wait();
    pdl_launch_dependents();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int m = p.m;
    const unsigned full = 0xffffffffu;
    if (staged)
        for (int i = tid; i < m; i += kSelThreads) ks[i] = p.key[i];
    const unsigned* keys = staged ? ks : p.key;
    if (tid == 0) {
        s_prefix = 0u;
        s_mask = 0u;
        s_rem = p.K;
    }
    for (int shift = 24; shift >= 0; shift -= 8) {
        if (tid < 256) hist[tid] = 0u;
        __syncthreads();
        const unsigned prefix = s_prefix, mask = s_mask;
        const int rem = s_rem;
        for (int base = 0; base < m; base += kSelThreads) {
            const int i = base + tid;
            unsigned dg = 256u;
            if (i < m) {
                const unsigned k = keys[i];
                if ((k & mask) == prefix) dg = (k >> shift) & 255u;
            }
            const unsigned peers = __match_any_sync(full, dg);
            if (dg < 256u && lane == __ffs(peers) - 1) atomicAdd(&hist[dg], (unsigned)__popc(peers));
        }
        __syncthreads();
        // the digit holding the rem-th largest key among those with the
        // prefix: inclusive counts from the top digit down
        unsigned c = 0u, inc = 0u;
        if (tid < 256) {
            c = hist[255 - tid];
            inc = c;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const unsigned n = __shfl_up_sync(full, inc, o);
                if (lane >= o) inc += n;
            }
            if (lane == 31) wsum[warp] = inc;
        }
        __syncthreads();
        if (tid < 256) {
            for (int w = 0; w < warp; ++w) inc += wsum[w];
            const unsigned exc = inc - c;
            if (exc < (unsigned)rem && (unsigned)rem <= inc) {
                s_prefix = prefix | ((255u - (unsigned)tid) << shift);
                s_mask = mask | (255u << shift);
                s_rem = rem - (int)exc;
            }
        }
        __syncthreads();
    }
    const unsigned T = s_prefix;
    const int need = s_rem;  // how many ids with key == T are kept

    const int span = ((m + kSelWarps - 1) / kSelWarps + 31) / 32 * 32;
    const int lo = min(m, warp * span), hi = min(m, lo + span);
    int gt = 0, eq = 0;
    for (int i0 = lo; i0 < hi; i0 += 32) {
        const int i = i0 + lane;
        const unsigned k = i < hi ? keys[i] : 0u;
        gt += __popc(__ballot_sync(full, i < hi && k > T));
        eq += __popc(__ballot_sync(full, i < hi && k == T));
    }
    if (lane == 0) {
        s_gt[warp] = gt;
        s_eq[warp] = eq;
    }
    __syncthreads();
    if (warp == 0) {
        int a = s_gt[lane], b = s_eq[lane];
        const int a0 = a, b0 = b;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int na = __shfl_up_sync(full, a, o), nb = __shfl_up_sync(full, b, o);
            if (lane >= o) {
                a += na;
                b += nb;
            }
        }
        s_gt[lane] = a - a0;
        s_eq[lane] = b - b0;
    }
    __syncthreads();
    int run_gt = s_gt[warp], run_eq = s_eq[warp];
    const unsigned below = (1u << lane) - 1u;
    for (int i0 = lo; i0 < hi; i0 += 32) {
        const int i = i0 + lane;
        const unsigned k = i < hi ? keys[i] : 0u;
        const bool is_gt = i < hi && k > T, is_eq = i < hi && k == T;
        const unsigned bg = __ballot_sync(full, is_gt), be = __ballot_sync(full, is_eq);
        const int eq_before = run_eq + __popc(be & below);
        const int pos = run_gt + __popc(bg & below) + min(eq_before, need);
        if ((is_gt || (is_eq && eq_before < need)) && pos < p.K) p.list[pos] = i;
        run_gt += __popc(bg);
        run_eq += __popc(be);
    }
}

// Exclusive prefix sums over the block's threads (thread order) of two
// counts at once, and their totals. Whole block; s_a, s_b hold kSelWarps ints.
__device__ __forceinline__ void block_scan2(int a, int b, int& ea, int& eb, int& ta, int& tb, int* s_a, int* s_b,
                                            int* s_tot) {
    const unsigned full = 0xffffffffu;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int ia = a, ib = b;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int na = __shfl_up_sync(full, ia, o), nb = __shfl_up_sync(full, ib, o);
        if (lane >= o) {
            ia += na;
            ib += nb;
        }
    }
    if (lane == 31) {
        s_a[warp] = ia;
        s_b[warp] = ib;
    }
    __syncthreads();
    if (warp == 0) {
        int wa = s_a[lane], wb = s_b[lane];
        const int wa0 = wa, wb0 = wb;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int na = __shfl_up_sync(full, wa, o), nb = __shfl_up_sync(full, wb, o);
            if (lane >= o) {
                wa += na;
                wb += nb;
            }
        }
        s_a[lane] = wa - wa0;
        s_b[lane] = wb - wb0;
        if (lane == 31) {
            s_tot[0] = wa;
            s_tot[1] = wb;
        }
    }
    __syncthreads();
    ea = s_a[warp] + ia - a;
    eb = s_b[warp] + ib - b;
    ta = s_tot[0];
    tb = s_tot[1];
    __syncthreads();  // s_a, s_b, s_tot may be reused
}

// The same selection for m <= kSelThreads * kSelKeys, led by the score
// kernel's histogram of the keys' top 12 bits. Thread t holds ids
// t*per .. t*per+per-1 in registers, so thread order is id order.
//   1. Thread t sums the copies of bins 4095-4t .. 4092-4t (highest first); a block scan
//      of their counts finds the bin B holding the K-th largest key and the
//      number of keys above it.
//   2. The keys in bin B (usually a few hundred) are compacted into shared
//      memory, and the (K - above)-th largest of their low 20 bits is found
//      digit by digit from the top (8, 8, then 4 bits: a shared histogram of
//      the next digit among the candidates matching the digits so far),
//      which gives the K-th largest key T.
//   3. A block scan of the per-thread counts of keys > T and == T places
//      every kept id in ascending order.
// Absent ids hold key 0 and are never counted.
constexpr int kSelKeys = 16;

// kSelThreads threads; cand: [m] unsigned of shared memory. Keys and the
// histogram are read at L2 (other CTAs may have just written them).
__device__ void select_hist_body(const PredictLaunch& p, unsigned* cand) {
    __shared__ int s_a[kSelWarps], s_b[kSelWarps], s_tot[2];
    __shared__ unsigned s_dig[256], s_sel[2];
    __shared__ int s_bin, s_above;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int m = p.m, K = p.K;
    const unsigned full = 0xffffffffu;
    const int per = (m + kSelThreads - 1) / kSelThreads;  // <= kSelKeys
    const int i0 = tid * per;
    unsigned key[kSelKeys];
#pragma unroll
    for (int q = 0; q < kSelKeys; ++q) key[q] = (q < per && i0 + q < m) ? __ldcg(p.key + i0 + q) : 0u;
    constexpr int BPT = kPredHistBins / kSelThreads;  // bins per thread
    int hv[BPT], hsum = 0;
#pragma unroll
    for (int q = 0; q < BPT; ++q) {
        hv[q] = 0;
#pragma unroll
        for (int part = 0; part < kPredHistParts; ++part)
            hv[q] += (int)__ldcg(p.hist + part * kPredHistBins + kPredHistBins - 1 - (BPT * tid + q));
        hsum += hv[q];
    }
    int above, unused, htot, unused2;
    block_scan2(hsum, 0, above, unused, htot, unused2, s_a, s_b, s_tot);
#pragma unroll
    for (int q = 0; q < BPT; ++q) {
        if (above < K && K <= above + hv[q]) {  // exactly one bin of one thread
            s_bin = kPredHistBins - 1 - (BPT * tid + q);
            s_above = above;
        }
        above += hv[q];
    }
    __syncthreads();
    const unsigned B = (unsigned)s_bin;
    const int need_in_bin = K - s_above;

    int c = 0;
#pragma unroll
    for (int q = 0; q < kSelKeys; ++q) c += (key[q] != 0u && (key[q] >> 20) == B) ? 1 : 0;
    int off, unused3, n_c, unused4;
    block_scan2(c, 0, off, unused3, n_c, unused4, s_a, s_b, s_tot);
#pragma unroll
    for (int q = 0; q < kSelKeys; ++q)
        if (key[q] != 0u && (key[q] >> 20) == B) cand[off++] = key[q] & 0xfffffu;
    __syncthreads();

    // the need_in_bin-th largest of the candidates' low 20 bits, by digits of
    // 8, 8 and 4 bits from the top: count the candidates that match the
    // digits found so far into a histogram of the next digit, then take the
    // digit holding the remaining rank (counting from the top)
    unsigned L = 0u, Lmask = 0u;
    int rem = need_in_bin;
    for (int pass = 0; pass < 3; ++pass) {
        const int shift = pass == 0 ? 12 : (pass == 1 ? 4 : 0);
        const int nb = pass == 2 ? 16 : 256;
        for (int i = tid; i < 256; i += kSelThreads) s_dig[i] = 0u;
        __syncthreads();
        for (int i = tid; i < n_c; i += kSelThreads) {
            const unsigned cv = cand[i];
            if ((cv & Lmask) == L) atomicAdd(&s_dig[(cv >> shift) & (unsigned)(nb - 1)], 1u);
        }
        __syncthreads();
        if (warp == 0) {
            // lane l holds the counts of digits nb-1-8l .. nb-8-8l (highest first)
            unsigned c8[8], sum = 0u;
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const int dgt = nb - 1 - 8 * lane - q;
                c8[q] = dgt >= 0 ? s_dig[dgt] : 0u;
                sum += c8[q];
            }
            unsigned incl = sum;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const unsigned nv = __shfl_up_sync(full, incl, o);
                if (lane >= o) incl += nv;
            }
            unsigned above_l = incl - sum;
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                if (above_l < (unsigned)rem && (unsigned)rem <= above_l + c8[q]) {
                    s_sel[0] = (unsigned)(nb - 1 - 8 * lane - q);
                    s_sel[1] = (unsigned)rem - above_l;
                }
                above_l += c8[q];
            }
        }
        __syncthreads();
        L |= s_sel[0] << shift;
        Lmask |= (unsigned)(nb - 1) << shift;
        rem = (int)s_sel[1];
        __syncthreads();  // s_dig and s_sel are rewritten by the next pass
    }
    const unsigned T = (B << 20) | L;

    int gt = 0, eq = 0;
#pragma unroll
    for (int q = 0; q < kSelKeys; ++q) {
        gt += (key[q] != 0u && key[q] > T) ? 1 : 0;
        eq += (key[q] != 0u && key[q] == T) ? 1 : 0;
    }
    int run_gt, run_eq, total_gt, total_eq;
    block_scan2(gt, eq, run_gt, run_eq, total_gt, total_eq, s_a, s_b, s_tot);
    const int need = K - total_gt;  // ids with key == T that are kept (the first ones)
#pragma unroll
    for (int q = 0; q < kSelKeys; ++q) {
        const unsigned k = key[q];
        if (k == 0u) continue;
        if (k > T) {
            p.list[run_gt + min(run_eq, need)] = i0 + q;
            ++run_gt;
        } else if (k == T) {
            if (run_eq < need) p.list[run_gt + run_eq] = i0 + q;
            ++run_eq;
        }
    }
}

__global__ void __launch_bounds__(kSelThreads) k_pred_select_hist(const PredictLaunch p) {
    extern __shared__ unsigned cand[];  // [m] low 20 bits of the keys in bin B
    pdl_wait();
    pdl_launch_dependents();
    select_hist_body(p, cand);
}

template <typename T, int NB>
cudaError_t launch_nb(const PredictLaunch& p, cudaLaunchConfig_t lc) {
    constexpr int N = Vec<T>::N;
    lc.gridDim = dim3(p.hid_grid);
    lc.blockDim = dim3(kPredThreads);
    lc.dynamicSmemBytes = (size_t)NB * p.d * sizeof(float);
    cudaError_t e = cudaLaunchKernelEx(&lc, k_pred_hidden<T, NB>, p);
    if (e != cudaSuccess) return e;
    lc.gridDim = dim3(p.score_grid);
    lc.dynamicSmemBytes = (size_t)NB * p.r * sizeof(float);
    switch (p.r / (kWarp * N)) {
        case 1: e = cudaLaunchKernelEx(&lc, k_pred_score<T, NB, 1>, p); break;
        case 2: e = cudaLaunchKernelEx(&lc, k_pred_score<T, NB, 2>, p); break;
        case 4: e = cudaLaunchKernelEx(&lc, k_pred_score<T, NB, 4>, p); break;
        case 8: e = cudaLaunchKernelEx(&lc, k_pred_score<T, NB, 8>, p); break;
        default: return cudaErrorInvalidValue;
    }
    if (e != cudaSuccess) return e;
    lc.gridDim = dim3(1);
    lc.blockDim = dim3(kSelThreads);
    if (p.m <= kSelThreads * kSelKeys) {
        lc.dynamicSmemBytes = (size_t)p.m * sizeof(unsigned);
        return cudaLaunchKernelEx(&lc, k_pred_select_hist, p);
    }
    const int staged = (size_t)p.m * sizeof(unsigned) <= (size_t)g_sel_smem;
    lc.dynamicSmemBytes = staged ? (size_t)p.m * sizeof(unsigned) : 0;
    return cudaLaunchKernelEx(&lc, k_pred_select, p, staged);
}

template <typename T>
cudaError_t launch_t(const PredictLaunch& p, cudaLaunchConfig_t lc) {
    switch (pow2_batch(p.batch)) {
        case 1: return launch_nb<T, 1>(p, lc);
        case 2: return launch_nb<T, 2>(p, lc);
        case 4: return launch_nb<T, 4>(p, lc);
        default: return launch_nb<T, 8>(p, lc);
    }
}

template <typename T, int NB>
cudaError_t prepare_nb(int optin_smem) {
    // static shared memory (the norm's reduction array) counts against the opt-in limit
    cudaError_t e = cudaFuncSetAttribute(k_pred_hidden<T, NB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         optin_smem - kSmemSlack);
    const int score_smem = NB * 8 * kWarp * Vec<T>::N * (int)sizeof(float);
    const cudaFuncAttribute a = cudaFuncAttributeMaxDynamicSharedMemorySize;
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_pred_score<T, NB, 1>, a, score_smem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_pred_score<T, NB, 2>, a, score_smem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_pred_score<T, NB, 4>, a, score_smem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_pred_score<T, NB, 8>, a, score_smem);
    return e;
}

template <typename T>
cudaError_t prepare_t(int optin_smem) {
    cudaError_t e = prepare_nb<T, 1>(optin_smem);
    if (e == cudaSuccess) e = prepare_nb<T, 2>(optin_smem);
    if (e == cudaSuccess) e = prepare_nb<T, 4>(optin_smem);
    if (e == cudaSuccess) e = prepare_nb<T, 8>(optin_smem);
    return e;
}

}  // namespace

bool predict_supported(int elem_bytes, int d, int r, int batch, int optin_smem) {
    if (elem_bytes != 2 && elem_bytes != 4) return false;
    const int per_warp = kWarp * (16 / elem_bytes);  // elements per 16-byte-per-lane step
    if (d < per_warp || r < per_warp || d % per_warp != 0 || r % per_warp != 0) return false;
    const int steps = r / per_warp;
    if (steps != 1 && steps != 2 && steps != 4 && steps != 8) return false;
    if (batch < 1 || batch > kPredMaxBatch) return false;
    return (size_t)pow2_batch(batch) * d * sizeof(float) + kSmemSlack <= (size_t)optin_smem;
}

void predict_geometry(PredictLaunch* p, int elem_bytes, int num_sms) {
    const int per_warp = kWarp * (16 / elem_bytes);
    const int steps = p->d / per_warp;
    int splits = 1;
    while (splits * 2 <= kPredMaxSplits && steps % (splits * 2) == 0 && steps / (splits * 2) >= 8 &&
           p->r * splits < num_sms * kPredWarps)
        splits *= 2;
    p->splits = splits;
    const int pieces = p->r * splits;
    p->hid_grid = std::max(1, std::min((pieces + kPredWarps - 1) / kPredWarps, 2 * num_sms));
    const int rsteps = p->r / per_warp;
    const int rg = rsteps >= 8 ? 1 : 8 / rsteps;
    const int groups = (p->m + rg - 1) / rg;
    p->score_grid = std::max(1, std::min((groups + kPredWarps - 1) / kPredWarps, 4 * num_sms));
}

cudaError_t prepare_predict(int optin_smem) {
    cudaError_t e = prepare_t<float>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<__nv_bfloat16>(optin_smem);
    const int sel_smem = std::min(kSelSmemMax, optin_smem - kSmemSlack);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_pred_select, cudaFuncAttributeMaxDynamicSharedMemorySize, sel_smem);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_pred_select_hist, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kSelThreads * kSelKeys * (int)sizeof(unsigned));
    if (e == cudaSuccess) g_sel_smem = sel_smem;
    return e;
}

cudaError_t launch_predict(const PredictLaunch& p, int elem_bytes, cudaStream_t stream, bool pdl) {
    cudaLaunchConfig_t lc = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = pdl ? 1 : 0;
    lc.stream = stream;
    return elem_bytes == 2 ? launch_t<__nv_bfloat16>(p, lc) : launch_t<float>(p, lc);
}

}  // namespace tsffn
