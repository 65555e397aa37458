// ts_kernels.cuh -- device helpers and launch parameter blocks shared by the
// sm_103a kernels of libtsffn (gate+up, down, router) and the C-ABI layer.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <type_traits>

namespace tsffn {

constexpr int kWarp = 32;
constexpr int kChunk = 8;       // rows per gate/up work item (one bitmap byte)
constexpr int kMaxPass = 8;     // tokens per pass of the CUDA-core kernels
constexpr int kMaxBatch = 64;   // largest dense batch
constexpr int kMaxMoeBatch = 8; // largest MoE batch
constexpr int kMaxExperts = 16;
constexpr int kMaxTopK = 4;
constexpr int kDownWarps = 16;
// Passes of at most this many tokens fold the down projection into the
// gate+up kernel (an accumulator warp per CTA writes a partial y) and finish
// it with a reduction over the CTAs' partials; wider passes gather W_down rows
// in a separate kernel.
constexpr int kAccMaxTokens = 2;
constexpr int kRouterMaxD = 16384;  // router keeps one fp32 activation row in shared memory

// device status bits (OR-ed into the handle's status word)
constexpr unsigned kStatusBadIndex = 1u;
constexpr unsigned kStatusTimeout = 2u;

// Gather-index checks of the debug build (compiled with -DTS_DEBUG): every row
// index a kernel is about to gather is compared with the row count m; a bad one
// is recorded as kStatusBadIndex in the status word and replaced by row 0, so
// the kernel stays in bounds. The release build validates the caller's lists
// once, where it reads them, and compiles these checks out.
#ifdef TS_DEBUG
__device__ __forceinline__ int debug_row(int j, int m, unsigned* status) {
    if ((unsigned)j < (unsigned)m) return j;
    atomicOr(status, kStatusBadIndex);
    return 0;
}
#else
__device__ __forceinline__ int debug_row(int j, int, unsigned*) { return j; }
#endif
// Bound on any device-side wait: a wait that lasts longer records
// kStatusTimeout and the kernel winds down instead of hanging.
constexpr unsigned long long kWaitLimitNs = 1000000000ull;

// Routing of one token: experts in selection order and their weights.
struct TokenRoute {
    int sel[kMaxTopK];
    float w[kMaxTopK];
};

// Per-expert (or the single FFN's) weight rows, [m][d] neuron-major.
struct ExpertPtrs {
    const void* wg;
    const void* wu;
    const void* wd;
};

// Parameters of one gate+up launch (K1+K2 fused) and the matching down
// launch (K3). A batch slot is the pass-local token (single FFN) or the
// global token (MoE). `route == nullptr` means a single FFN whose experts[0] gets the
// pass's tokens tok0 .. tok0+nt-1 with weight 1.
struct FfnLaunch {
    int d, m;
    int elem_bytes;         // bytes per weight element (2 bf16, 4 fp32; 0 for INT4 rows)
    int row_bytes;          // bytes per weight row (d * elem_bytes, or 9d/16 for INT4)
    int n_rows;             // size of the row space: m, or the list length
    const int32_t* rows;    // predictor list (ascending neuron ids) or nullptr
    int batch;              // tokens of the whole call
    int tok0, nt;           // this pass: tokens tok0 .. tok0+nt-1 (dense only)
    const void* x;          // [batch][d] activations, weight dtype
    float* h;               // [batch][d] residual (stack mode) or nullptr
    float* y;               // [batch][d] output (forward mode)
    int norm_from_h;        // 1: x = rmsnorm(h) computed in the gate+up prologue
    int n_experts;
    ExpertPtrs ex[kMaxExperts];
    const TokenRoute* route;  // MoE routing [batch] or nullptr
    int top_k;
    // scratch
    float* cval;            // [expert][batch slot][n_rows_cap]: routed w * c at union rows
    int cval_tok_stride;    // n_rows_cap
    uint8_t* gbits;         // per-token gate-active bitmap bytes
    uint8_t* bbits;         // per-token both-active bitmap bytes
    long long bits_expert_stride;  // bytes between experts (0 for a single FFN)
    int bits_tok_base;      // token index of local token 0 in the bitmaps (tok0 for dense)
    int nbytes;             // bitmap bytes per token (multiple of 4)
    uint8_t* ubits;         // [expert][nbytes] union over the pass's tokens: both-active
    uint8_t* ugbits;        // [expert][nbytes] union gate-active
    unsigned* status;
    int residual_out;       // 1: h += y instead of y =
    // Partial down projections of passes of <= kAccMaxTokens tokens,
    // [gate+up CTA][partial_slots][d] fp32: gate+up CTA b writes slots
    // 0 .. n_slots-1 of block b; the reduction sums blocks 0 .. partial_ctas-1.
    float* partial;
    int partial_slots;
    int partial_ctas;
    // Test hook (failure detection): nonzero makes consumer warp 0 of every
    // gate+up CTA wait on a barrier nothing arrives at, so the bounded wait
    // runs out and the status word records kStatusTimeout.
    int test_stall;
    // Nonzero when `rows` (the predictor list) was written before the
    // kernels preceding this launch in the stream ran, so it may be read
    // before waiting for them (stack layers after the first, with the
    // caller's lists).
    int rows_ready;
    // Nonzero when the residual h (stack mode) was final before the kernels
    // preceding this launch in the stream ran (the predicted stack: the
    // predictor's kernels sit between the last writer of h and this launch),
    // so the activations may be staged before waiting for them.
    int h_ready;
    // Nonzero when the kernel after this launch's reduction is the next
    // layer's first kernel in an FFN stack (its gate+up kernel, or the
    // predictor's first kernel): the reduction lets it be scheduled before
    // its own wait. (The MoE stack, whose router comes next, measured slower
    // so.)
    int trigger_early;
    // Stack mode: the next layer's W_gate (nullptr: none), its row count and
    // its gate+up grid. The gathered down kernel (passes of 4-8 tokens),
    // before waiting for the gate+up kernel, prefetches into L2 the first
    // prefetch_rows rows each next-layer gate+up CTA will stream, so HBM keeps
    // working while this layer's up rows and down projection finish.
    const void* next_wg;
    int next_n_rows;
    int next_grid;
    int prefetch_rows;
};

// The fused layer stack (passes of 1-2 tokens, bf16 rows, single FFNs): one
// cooperative launch runs every layer's gate+up, down partial and reduction,
// with grid barriers between the dependent steps instead of kernel
// boundaries.
struct StackLaunch {
    const FfnLaunch* layers;  // device array [n_layers]; each layer's own scratch
    int n_layers;
    float* h;                 // [nt][d] residual, updated in place
    unsigned* bar;            // zero before the launch: barrier counters and abort flag (stack_bar_words)
    unsigned* status;         // barrier timeouts are recorded here
};

struct RouterLaunch {
    int d, n_experts, top_k, batch;
    const void* x;          // [batch][d] or nullptr in norm mode
    const float* h;         // [batch][d] residual (norm mode)
    void* xbuf;             // [batch][d] normalised activations written in norm mode
    const void* wr;         // [n_experts][d]
    TokenRoute* route;      // [batch] out
};

// ---------------------------------------------------------------------------
// device helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 ld_stream(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// Programmatic dependent launch: wait for the previous grid's results / let
// the next grid start its independent prologue.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Asynchronous L2 prefetch of `bytes` (multiple of 16) at a 16-byte aligned address.
__device__ __forceinline__ void prefetch_l2_bulk(const void* p, unsigned bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// ---- shared-memory barriers and 1-D bulk copies (TMA) ----------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, unsigned count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_fence_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, unsigned bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}
// Raise the transaction count the current phase waits for, without arriving.
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, unsigned bytes) {
    asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, unsigned parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// As mbar_try_wait, but a waiting thread is suspended (it stops issuing)
// until the phase completes or about `hint_ns` pass.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t* bar, unsigned parity, unsigned hint_ns) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "r"(hint_ns)
        : "memory");
    return ok != 0;
}
// Wait for the phase with the given parity to complete, for at most
// kWaitLimitNs; false on timeout (the caller records it and winds down).
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, unsigned parity) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    while (!mbar_try_wait_sleep(bar, parity, 1000000u))
        if (global_ns() - t0 > kWaitLimitNs) return false;
    return true;
}
// Order this thread's earlier generic-proxy accesses to shared memory before
// its later async-proxy (bulk copy) accesses, e.g. reads of a slot before a
// copy that overwrites it.
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// 1-D bulk copy global -> this CTA's shared memory, completing on `bar`.
__device__ __forceinline__ void tma_load_1d(void* dst, const void* src, unsigned bytes, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}
__device__ __forceinline__ uint4 lds128(const void* p) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(smem_u32(p)));
    return v;
}
__device__ __forceinline__ void named_bar_sync(int id, int threads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Elements of a 16-byte vector, as fp32.
template <typename T>
struct Vec;

template <>
struct Vec<float> {
    static constexpr int N = 4;
    __device__ __forceinline__ static void unpack(const uint4& v, float* o) {
        o[0] = __uint_as_float(v.x);
        o[1] = __uint_as_float(v.y);
        o[2] = __uint_as_float(v.z);
        o[3] = __uint_as_float(v.w);
    }
    __device__ __forceinline__ static float load1(const void* p, size_t i) {
        return static_cast<const float*>(p)[i];
    }
    __device__ __forceinline__ static float round_act(float v) { return v; }
    __device__ __forceinline__ static void store1(void* p, size_t i, float v) {
        static_cast<float*>(p)[i] = v;
    }
};

template <>
struct Vec<__nv_bfloat16> {
    static constexpr int N = 8;
    __device__ __forceinline__ static void unpack(const uint4& v, float* o) {
        o[0] = bf16lo(v.x); o[1] = bf16hi(v.x);
        o[2] = bf16lo(v.y); o[3] = bf16hi(v.y);
        o[4] = bf16lo(v.z); o[5] = bf16hi(v.z);
        o[6] = bf16lo(v.w); o[7] = bf16hi(v.w);
    }
    __device__ __forceinline__ static float load1(const void* p, size_t i) {
        return __bfloat162float(static_cast<const __nv_bfloat16*>(p)[i]);
    }
    __device__ __forceinline__ static float round_act(float v) {
        return __bfloat162float(__float2bfloat16_rn(v));
    }
    __device__ __forceinline__ static void store1(void* p, size_t i, float v) {
        static_cast<__nv_bfloat16*>(p)[i] = __float2bfloat16_rn(v);
    }
};

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Expert/token bookkeeping resolved by every CTA from the routing table.
struct ExpertSets {
    int n_act;                          // experts with at least one token
    int act[kMaxExperts];               // their ids, ascending
    int ntok[kMaxExperts];              // tokens per expert
    int tok[kMaxExperts][kMaxMoeBatch];  // global token ids, ascending
    float w[kMaxExperts][kMaxMoeBatch];  // routing weights
};

// Fill `s` (shared memory) from the launch; call with the whole block, ends
// with __syncthreads(). Single FFN: one expert with tokens tok0..tok0+nt-1.
__device__ __forceinline__ void resolve_experts(const FfnLaunch& a, ExpertSets& s) {
    if (threadIdx.x < kWarp) {
        const int lane = threadIdx.x;
        if (a.route == nullptr) {
            if (lane == 0) {
                s.n_act = 1;
                s.act[0] = 0;
                s.ntok[0] = a.nt;
            }
            if (lane < a.nt) {
                s.tok[0][lane] = a.tok0 + lane;
                s.w[0][lane] = 1.0f;
            }
        } else {
            // lane e collects the tokens routed to expert e, in token order
            int n = 0;
            if (lane < a.n_experts) {
                for (int t = 0; t < a.batch; ++t) {
                    const TokenRoute r = a.route[t];
                    for (int k = 0; k < a.top_k; ++k) {
                        if (r.sel[k] == lane && n < kMaxMoeBatch) {
                            s.tok[lane][n] = t;
                            s.w[lane][n] = r.w[k];
                            ++n;
                        }
                    }
                }
                s.ntok[lane] = n;
            }
            const unsigned has = __ballot_sync(0xffffffffu, lane < a.n_experts && n > 0);
            if (lane < a.n_experts && n > 0) s.act[__popc(has & ((1u << lane) - 1u))] = lane;
            if (lane == 0) s.n_act = __popc(has);
        }
    }
    __syncthreads();
}

// One activation row of a gate+up CTA's consumer threads (ctid < cthreads,
// cwarp = ctid / 32, named barrier 1), handed element by element to
// put(i, v): x = round(h / sqrt(mean(h^2) + 1e-5)) with x[d-1] = 1 when
// `h` is given (stack mode), else the row of x as stored. Every global load
// of a group of kStageVec 16-byte vectors per thread is issued before any is
// used, so the row arrives in one memory round trip instead of one per
// element; for d <= 4 * kStageVec * cthreads the h values stay in registers
// between the sum of squares and the division. The sum of squares runs in a
// fixed order (per thread, then the warp tree, then warps in order), so every
// CTA computes the same bits. `red` holds one float per consumer warp.
// `after_loads()` runs once, right after the first group's loads are
// issued and before any of them is used: work placed there (such as the
// first weight-row copies) queues behind the activations instead of ahead.
constexpr int kStageVec = 4;

struct NoAfterLoads {
    __device__ __forceinline__ void operator()() const {}
};

template <typename T, typename Put, typename After = NoAfterLoads>
__device__ __forceinline__ void stage_act_row(const float* __restrict__ h, const void* x, int d, int ctid,
                                              int cthreads, float* red, Put put, After after_loads = After()) {
    const int lane = ctid & 31, cwarp = ctid >> 5, nw = cthreads >> 5;
    if (h != nullptr) {
        const bool vec = (d % 4) == 0 && (reinterpret_cast<uintptr_t>(h) & 15u) == 0;
        const int d4 = vec ? d / 4 : 0;
        const int group = kStageVec * cthreads;  // float4 per group
        float4 v[kStageVec];
        float ss = 0.0f;
        if (d4 == 0) after_loads();
        for (int g0 = 0; g0 < d4; g0 += group) {
#pragma unroll
            for (int k = 0; k < kStageVec; ++k) {
                const int q = g0 + ctid + k * cthreads;
                v[k] = q < d4 ? __ldcg(reinterpret_cast<const float4*>(h + 4 * (size_t)q)) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
            if (g0 == 0) after_loads();
#pragma unroll
            for (int k = 0; k < kStageVec; ++k) {
                ss = fmaf(v[k].x, v[k].x, ss);
                ss = fmaf(v[k].y, v[k].y, ss);
                ss = fmaf(v[k].z, v[k].z, ss);
                ss = fmaf(v[k].w, v[k].w, ss);
            }
        }
        for (int i = 4 * d4 + ctid; i < d; i += cthreads) ss = fmaf(h[i], h[i], ss);  // rows with d % 4 != 0
        ss = warp_sum(ss);
        if (lane == 0) red[cwarp] = ss;
        named_bar_sync(1, cthreads);
        float tot = 0.0f;
        for (int w = 0; w < nw; ++w) tot += red[w];
        const float rms = __fsqrt_rn(__fadd_rn(__fdiv_rn(tot, (float)d), 1e-5f));
        const float rinv = __frcp_rn(rms);  // one reciprocal, then a product per element
        auto norm = [&](int i, float hv) { return (i == d - 1) ? 1.0f : Vec<T>::round_act(__fmul_rn(hv, rinv)); };
        const bool kept = d4 <= group;  // the single group is still in registers
        for (int g0 = 0; g0 < d4; g0 += group) {
#pragma unroll
            for (int k = 0; k < kStageVec; ++k) {
                const int q = g0 + ctid + k * cthreads;
                if (q < d4) {
                    const float4 w = kept ? v[k] : __ldcg(reinterpret_cast<const float4*>(h + 4 * (size_t)q));
                    if constexpr (std::is_invocable_v<Put, int, float4>) {
                        // elements 4q .. 4q + 3 in one store
                        put(4 * q, make_float4(norm(4 * q, w.x), norm(4 * q + 1, w.y), norm(4 * q + 2, w.z),
                                               norm(4 * q + 3, w.w)));
                    } else {
                        put(4 * q, norm(4 * q, w.x));
                        put(4 * q + 1, norm(4 * q + 1, w.y));
                        put(4 * q + 2, norm(4 * q + 2, w.z));
                        put(4 * q + 3, norm(4 * q + 3, w.w));
                    }
                }
            }
        }
        for (int i = 4 * d4 + ctid; i < d; i += cthreads) put(i, norm(i, h[i]));
        named_bar_sync(1, cthreads);  // red[] is reused by the next row
    } else {
        constexpr int N = Vec<T>::N;  // elements per 16-byte vector
        const bool vec = (d % N) == 0 && (reinterpret_cast<uintptr_t>(x) & 15u) == 0;
        const int dv = vec ? d / N : 0;
        const int group = kStageVec * cthreads;
        if (dv == 0) after_loads();
        for (int g0 = 0; g0 < dv; g0 += group) {
            uint4 w[kStageVec];
#pragma unroll
            for (int k = 0; k < kStageVec; ++k) {
                const int q = g0 + ctid + k * cthreads;
                w[k] = q < dv ? *reinterpret_cast<const uint4*>(static_cast<const unsigned char*>(x) + 16 * (size_t)q)
                              : make_uint4(0u, 0u, 0u, 0u);
            }
            if (g0 == 0) after_loads();
#pragma unroll
            for (int k = 0; k < kStageVec; ++k) {
                const int q = g0 + ctid + k * cthreads;
                if (q < dv) {
                    float f[N];
                    Vec<T>::unpack(w[k], f);
#pragma unroll
                    for (int e = 0; e < N; ++e) put(N * q + e, f[e]);
                }
            }
        }
        for (int i = N * dv + ctid; i < d; i += cthreads) put(i, Vec<T>::load1(x, (size_t)i));
    }
}

// x = round(h / sqrt(mean(h^2) + 1e-5)), x[d-1] = 1, into shared memory, by
// the whole block (blockDim.x a multiple of 32, `red` one float per warp).
// Every block computes the same bits (fixed per-thread order, fixed tree).
template <typename T>
__device__ __forceinline__ void block_rmsnorm(const float* __restrict__ h, int d, float* __restrict__ out,
                                              float* red) {
    stage_act_row<T>(h, nullptr, d, (int)threadIdx.x, (int)blockDim.x, red, [&](int i, float v) { out[i] = v; });
    __syncthreads();
}

}  // namespace tsffn

// Host-side launchers (defined in the kernel translation units).
namespace tsffn {
cudaError_t launch_gate_up(const FfnLaunch& a, int wdtype, int pass_tokens, int grid,
                           cudaStream_t stream, bool pdl);
// Top-k magnitude mask (Eq. 3-4) on a pass's c values and both-active bitmaps.
cudaError_t launch_topk(const FfnLaunch& a, int keep, cudaStream_t stream);
cudaError_t launch_down(const FfnLaunch& a, int wdtype, int pass_tokens, cudaStream_t stream,
                        bool pdl);
// Sum of the gate+up CTAs' partial down projections (passes of <= kAccMaxTokens).
cudaError_t launch_down_reduce(const FfnLaunch& a, int pass_tokens, cudaStream_t stream, bool pdl);
cudaError_t launch_router(const RouterLaunch& a, int wdtype, cudaStream_t stream, bool pdl);
// Set per-kernel attributes once per device, before any launch or capture.
cudaError_t prepare_gate_up(int optin_smem);
cudaError_t prepare_down();
cudaError_t prepare_router();
// Ring geometry of the gate+up kernel for `x_tokens` activation rows in
// shared memory; -1 if fewer than 4 row slots fit.
int gate_up_config(int wdtype, int d, int x_tokens, int optin_smem, int* slots, int* slot_bytes,
                   int* xs_stride, size_t* smem);
// Whether INT4 rows of d weights can run passes of `pass_tokens` tokens.
bool int4_supported(int d, int pass_tokens, int optin_smem);
// The fused layer stack: whether a stack of bf16 layers of width d, passes of
// nt tokens (1-2), can run as one cooperative launch of `grid` CTAs; and the
// launch.
bool stack_fused_supported(int d, int nt, int grid, int optin_smem);
cudaError_t launch_stack_fused(const StackLaunch& S, int d, int nt, int grid, cudaStream_t stream);
// 32-bit words of StackLaunch::bar for a grid of `grid` CTAs.
int stack_bar_words(int grid);
}  // namespace tsffn
