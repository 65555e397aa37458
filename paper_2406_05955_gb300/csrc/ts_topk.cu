// ts_topk.cu -- the top-k magnitude mask of Eq. 3-4 between the gate+up and
// the down launches of a pass: per token, only the `keep` neurons with the
// largest |Combined| (Combined = max(0, g) max(0, u), Eq. 2; a lower neuron
// index wins a tie) keep their c; the down projection then sums
// (Combined * Mask) W_down. Candidates are the token's both-active rows (every
// other row has Combined = 0 and adds nothing whether kept or not).
#include "ts_kernels.cuh"

namespace tsffn {
namespace {

constexpr int kSelThreads = 1024;
constexpr int kSelWarps = kSelThreads / kWarp;
constexpr int kKeyCache = 8;  // candidate keys a thread keeps in shared memory (the rest are re-read)

// Exclusive prefix of v over the block in thread order, and the block total
// (warp shuffles, then one warp over the warp sums).
__device__ __forceinline__ int block_excl_scan(int v, int* s_warp, int* s_total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = v;
#pragma unroll
    for (int o = 1; o < kWarp; o <<= 1) {
        const int n = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += n;
    }
    if (lane == kWarp - 1) s_warp[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        const int w = lane < kSelWarps ? s_warp[lane] : 0;
        int wi = w;
#pragma unroll
        for (int o = 1; o < kWarp; o <<= 1) {
            const int n = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += n;
        }
        if (lane < kSelWarps) s_warp[lane] = wi - w;
        if (lane == kWarp - 1) *s_total = wi;
    }
    __syncthreads();
    const int r = s_warp[warp] + incl - v;
    __syncthreads();  // s_warp is reused by the next scan
    return r;
}

// One CTA per token of the pass. c > 0 at a both-active row, so the fp32 bit
// pattern orders the candidates; an MSB-first radix select (four 8-bit
// digits) finds the keep-th largest key T, then the rows with key > T and the
// first rows (ascending) with key == T are kept. Threads own contiguous byte
// ranges of the bitmap, so a block prefix over the threads is row order; each
// thread keeps its first kKeyCache candidate keys in shared memory for the
// passes.
__global__ void __launch_bounds__(kSelThreads) k_topk_select(const FfnLaunch a, int keep) {
    __shared__ unsigned hist[256];
    __shared__ unsigned s_key[kKeyCache * kSelThreads];  // [slot][thread]: a thread's first candidates
    __shared__ int s_warp[kSelWarps];
    __shared__ unsigned s_prefix, s_mask;
    __shared__ int s_remaining, s_total;
    pdl_wait();
    pdl_launch_dependents();
    const int k = blockIdx.x;  // batch slot of the pass
    const int tid = threadIdx.x;
    float* cv = a.cval + (size_t)k * a.cval_tok_stride;
    uint8_t* bb = a.bbits + (size_t)(a.bits_tok_base + k) * a.nbytes;
    const int n_bytes = (a.n_rows + 7) / 8;
    const int per = (n_bytes + kSelThreads - 1) / kSelThreads;
    const int b0 = min(tid * per, n_bytes), b1 = min(b0 + per, n_bytes);
    auto key_ld = [&](int p) { return __float_as_uint(cv[p]); };
    // the i-th candidate of this thread (row p): from shared memory for the
    // first kKeyCache, else from c
    auto key_of = [&](int i, int p) { return i < kKeyCache ? s_key[i * kSelThreads + tid] : key_ld(p); };

    // candidates, the first kKeyCache keys of each thread kept in shared memory
    int cnt = 0;
    for (int b = b0; b < b1; ++b)
        for (unsigned bits = bb[b]; bits; bits &= bits - 1u, ++cnt)
            if (cnt < kKeyCache) s_key[cnt * kSelThreads + tid] = key_ld(b * 8 + __ffs(bits) - 1);
    block_excl_scan(cnt, s_warp, &s_total);
    if (tid == 0) {
        s_prefix = 0u;
        s_mask = 0u;
        s_remaining = keep;
    }
    __syncthreads();
    if (keep >= s_total) return;  // every candidate is kept

    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int i = tid; i < 256; i += kSelThreads) hist[i] = 0u;
        __syncthreads();
        const unsigned prefix = s_prefix, mask = s_mask;
        int i = 0;
        for (int b = b0; b < b1; ++b)
            for (unsigned bits = bb[b]; bits; bits &= bits - 1u, ++i) {
                const unsigned key = key_of(i, b * 8 + __ffs(bits) - 1);
                if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
            }
        __syncthreads();
        if (tid < kWarp) {
            // the digit of the keep-th largest key among those with the
            // prefix: lane l holds digits 255 - 8l .. 248 - 8l, highest first
            const int lane = tid;
            const int rem0 = s_remaining;
            int c8[8], sum = 0;
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                c8[q] = (int)hist[255 - 8 * lane - q];
                sum += c8[q];
            }
            int incl = sum;
#pragma unroll
            for (int o = 1; o < kWarp; o <<= 1) {
                const int n = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += n;
            }
            int above = incl - sum;  // keys in higher digits
            // the highest digit whose count from the top reaches rem0 (digit
            // 0 when none does, as a scan from the top stops at the bottom)
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const int dg = 255 - 8 * lane - q;
                const bool reach = above + c8[q] >= rem0;
                const bool first = dg == 255 || above < rem0;
                if (first && (reach || dg == 0)) {
                    s_prefix = prefix | ((unsigned)dg << shift);
                    s_remaining = rem0 - above;  // how many keys equal to the final prefix are kept, at the end
                }
                above += c8[q];
            }
            if (lane == 0) s_mask = mask | (255u << shift);
        }
        __syncthreads();
    }
    const unsigned T = s_prefix;
    const int need_eq = s_remaining;
    // rank of each key == T in row order
    int eq = 0;
    {
        int i = 0;
        for (int b = b0; b < b1; ++b)
            for (unsigned bits = bb[b]; bits; bits &= bits - 1u, ++i) eq += key_of(i, b * 8 + __ffs(bits) - 1) == T;
    }
    int rank = block_excl_scan(eq, s_warp, &s_total);
    int i = 0;
    for (int b = b0; b < b1; ++b) {
        unsigned kept = 0u;
        for (unsigned bits = bb[b]; bits; bits &= bits - 1u, ++i) {
            const int r = __ffs(bits) - 1;
            const int p = b * 8 + r;
            const unsigned key = key_of(i, p);
            bool keep_it = key > T;
            if (key == T) keep_it = rank++ < need_eq;
            if (keep_it)
                kept |= 1u << r;
            else
                cv[p] = 0.0f;  // the down projection multiplies by c
        }
        bb[b] = (uint8_t)kept;
    }
}

// The pass's union both-active bytes from the masked per-token bytes.
__global__ void __launch_bounds__(256) k_topk_union(const FfnLaunch a) {
    pdl_wait();
    pdl_launch_dependents();
    const int n_bytes = (a.n_rows + 7) / 8;
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= n_bytes) return;
    unsigned u = 0u;
    for (int k = 0; k < a.nt; ++k) u |= a.bbits[(size_t)(a.bits_tok_base + k) * a.nbytes + b];
    a.ubits[b] = (uint8_t)u;
}

}  // namespace

cudaError_t launch_topk(const FfnLaunch& a, int keep, cudaStream_t stream) {
    cudaLaunchConfig_t lc = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = 1;
    lc.stream = stream;
    lc.gridDim = dim3(a.nt);
    lc.blockDim = dim3(kSelThreads);
    cudaError_t e = cudaLaunchKernelEx(&lc, k_topk_select, a, keep);
    if (e != cudaSuccess) return e;
    const int n_bytes = (a.n_rows + 7) / 8;
    lc.gridDim = dim3((n_bytes + 255) / 256);
    lc.blockDim = dim3(256);
    return cudaLaunchKernelEx(&lc, k_topk_union, a);
}

}  // namespace tsffn
