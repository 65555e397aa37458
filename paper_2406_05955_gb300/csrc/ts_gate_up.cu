// ts_gate_up.cu -- fused gate GEMV + ReLU + compaction and gathered up
// projection + dReLU product + second compaction (Eq. 1 with Eq. 2), for
// passes of up to 8 tokens. Every kernel is persistent, one CTA per SM, and
// works on items = (expert, chunk of kChunk consecutive rows of the row
// space), each CTA a contiguous range of items; W_up rows are read only for
// gate-active neurons, and each finished chunk's per-token bitmap bytes,
// union bytes and c = w_route * g * u are written out (finalize_chunks).
//   * k_gate_up_rows (bf16, 1-2 tokens, the decode path): no producer. Each
//     consumer warp copies its own rows with 16-byte cp.async into its own
//     ring slots, a few rows ahead of the one it computes; a round of chunks
//     is a gate phase (every gate row shared out one at a time), then an up
//     phase (every gate-active row), then the chunks are finalised; then the
//     CTA sums its both-active W_down rows into its block of the partial
//     buffer (down_partial), which k_down_reduce adds up over the CTAs.
//   * k_gate_up_q4w (INT4 rows, 1-2 tokens): the same rounds in subtasks of
//     4 rows, unpacked to bf16 in registers for mma.sync.
//   * k_gate_up_mma (bf16, 4-8 tokens): a producer thread fills a ring of
//     8-row groups with 1-D bulk copies; all consumer warps share each group
//     over K slices with mma.sync.
//   * k_gate_up (fp32, and bf16 where the others do not fit): a producer
//     thread fills a ring of whole-row slots, gate rows of chunk c then the
//     up rows of chunk c - kLookahead; consumers take slots round-robin.
//   * k_stack_rows: every layer of a batch-1-2 stack in one cooperative
//     launch, k_gate_up_rows's phases per layer with grid barriers around
//     the cross-CTA reduction.
// Where a kernel's rows do not depend on earlier kernels, it starts copying
// them before griddepcontrol.wait. Every wait on an mbarrier, a flag or the
// grid is bounded (kWaitLimitNs); on expiry the status word gets
// kStatusTimeout and the CTA drains its copies and returns.
#include <type_traits>

#include "ts_kernels.cuh"

namespace tsffn {

// consumer warps per CTA for NT tokens per pass; the ring's slot count is a
// multiple of it
template <int NT>
struct GateUpWarps {
    static constexpr int C = 8;
    static constexpr int THREADS = (C + 1) * kWarp;
};
constexpr int kMaxConsumers = 16;
constexpr int kWindow = 8;     // chunks in flight per CTA
constexpr int kLookahead = 3;  // gate chunks issued ahead of their up rows (< kWindow)
constexpr int kMaxSlots = 32;
constexpr int kRingBytes = 128 * 1024;  // ring budget: leaves room for down-projection CTAs
constexpr int kSmemMargin = 8192;       // static shared memory headroom

enum : int { kTaskGate = 0, kTaskUp = 1, kTaskEnd = 2 };

struct Task {
    int r;     // row within the chunk
    int cw;    // window slot of the chunk
    int kind;  // kTaskGate, kTaskUp, kTaskEnd
    int pad;
};

template <int NT>
struct ChunkState {
    int e, chunk, q, n_gate, gate_cnt, up_cnt;
    unsigned gmask;
    int jr[kChunk];
    float g[kChunk][NT];
    float u[kChunk][NT];
};

// Passes of <= kAccMaxTokens tokens: what the end-of-CTA down projection
// needs from each finished chunk (local index q < kMaxLocal; later chunks are
// read back from global memory), and the staging of its W_down rows.
constexpr int kMaxLocal = 32;
constexpr int kRoundCap = 48;  // rows listed per round
struct PartialShared {
    uint8_t ub[kMaxLocal];                         // both-active rows of chunk q
    float c[kMaxLocal][kChunk][kAccMaxTokens];     // their c values by batch slot
    const void* rowp[kRoundCap];                   // this round's rows: W_down row address
    float cs[kRoundCap][kAccMaxTokens];            // and c values
    int n_rows, next_item;                         // rows listed this round, first item of the next
};
struct NoPartial {};

template <int NT>
struct GateUpShared {
    typename std::conditional<(NT <= kAccMaxTokens), PartialShared, NoPartial>::type pd;
    uint64_t full[kMaxSlots];
    uint64_t empty[kMaxSlots];
    uint64_t gate_ready[kWindow];
    uint64_t chunk_free[kWindow];
    uint64_t never;  // nothing arrives here (FfnLaunch::test_stall)
    int mma_ok;      // tensor-core consumers: every wait so far succeeded
    Task task[kMaxSlots];
    ChunkState<NT> cs[kWindow];
    int q4_ctr[4];                 // INT4 kernel: subtasks claimed per phase, up subtasks
    unsigned q4_up[2 * kMaxLocal];  // INT4 kernel: up subtasks (chunk << 8 | rows)
    ExpertSets es;
    float red[kMaxConsumers];
};

struct GateUpCfg {
    int slots;       // ring slots S
    int slot_bytes;  // bytes per slot: one row, rounded up to 128
    int xs_stride;   // floats per activation row in shared memory (d rounded up to 256)
};

// Activation layout in shared memory: for bf16 rows each 256-element block is
// stored as [half h][lane l][4] for element l*8 + h*4 + q, so the two 16-byte
// reads of a lane hit consecutive addresses across the warp.
template <typename T>
__device__ __forceinline__ int xs_index(int i) {
    if (Vec<T>::N == 8)
        return (i & ~255) | (((i >> 2) & 1) << 7) | (((i >> 3) & 31) << 2) | (i & 3);
    return i;
}

// Writes staged activations into an fp32 row at xs_index positions: one
// element, or four consecutive ones (i a multiple of 4, which xs_index keeps
// contiguous and 16-byte aligned) in one store.
template <typename T>
struct XsPut {
    float* row;
    __device__ __forceinline__ void operator()(int i, float v) const { row[xs_index<T>(i)] = v; }
    __device__ __forceinline__ void operator()(int i, float4 v) const {
        *reinterpret_cast<float4*>(row + xs_index<T>(i)) = v;
    }
};

// acc[k] = sum_i row[i] * x_{xt[k]}[i] for k < ntok (row in shared memory).
// Each lane keeps ACC independent partial sums per token (element q of a
// 16-byte vector goes to sum q % ACC) so the FMAs do not form one serial
// dependency chain; the sums are combined before the warp reduction.
template <typename T, int NT>
__device__ __forceinline__ void smem_row_dot(const unsigned char* row, const float* xs, int xs_stride,
                                             const int (&xt)[NT], int ntok, int d, int lane,
                                             float (&acc)[NT]) {
    constexpr int VEC = Vec<T>::N;
    constexpr int BLK = kWarp * VEC;
    constexpr int ACC = NT >= 8 ? 1 : (NT == 4 ? 2 : (NT == 2 ? 4 : VEC));
    float part[NT][ACC];
    const float* xr[NT];
#pragma unroll
    for (int k = 0; k < NT; ++k) {
        xr[k] = xs + (size_t)xt[k] * xs_stride + (VEC == 8 ? lane * 4 : 0);
#pragma unroll
        for (int q = 0; q < ACC; ++q) part[k][q] = 0.0f;
    }
#pragma unroll 4
    for (int col = lane * VEC; col < d; col += BLK) {
        float f[VEC];
        Vec<T>::unpack(lds128(row + (size_t)col * sizeof(T)), f);
#pragma unroll
        for (int k = 0; k < NT; ++k) {
            if (NT == 1 || k < ntok) {
                const float* xk = xr[k];
                float xv[VEC];
                if (VEC == 8) {
                    const int xb = col & ~(BLK - 1);
                    const uint4 x0 = lds128(xk + xb);
                    const uint4 x1 = lds128(xk + xb + 128);
                    xv[0] = __uint_as_float(x0.x); xv[1] = __uint_as_float(x0.y);
                    xv[2] = __uint_as_float(x0.z); xv[3] = __uint_as_float(x0.w);
                    xv[4 % VEC] = __uint_as_float(x1.x); xv[5 % VEC] = __uint_as_float(x1.y);
                    xv[6 % VEC] = __uint_as_float(x1.z); xv[7 % VEC] = __uint_as_float(x1.w);
                } else {
                    const uint4 x0 = lds128(xk + col);
                    xv[0] = __uint_as_float(x0.x); xv[1] = __uint_as_float(x0.y);
                    xv[2 % VEC] = __uint_as_float(x0.z); xv[3 % VEC] = __uint_as_float(x0.w);
                }
#pragma unroll
                for (int q = 0; q < VEC; ++q) part[k][q % ACC] = fmaf(f[q], xv[q], part[k][q % ACC]);
            }
        }
    }
#pragma unroll
    for (int k = 0; k < NT; ++k) {
        float s = 0.0f;
#pragma unroll
        for (int q = 0; q < ACC; ++q) s += part[k][q];
        acc[k] = warp_sum(s);
    }
}

// Warp-wide: lane 0 waits on `bar`, every lane learns the outcome.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, unsigned parity, int lane, unsigned* status) {
    int ok = 1;
    if (lane == 0) {
        ok = mbar_wait(bar, parity) ? 1 : 0;
        if (!ok) atomicOr(status, kStatusTimeout);
    }
    return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

// Write finished chunks' outputs: per-token gate/both bitmap bytes, union
// bytes, and c by batch slot. One warp takes up to kWarp / kChunk chunks at
// once, chunk tab[c0 + q] in lanes 8q .. 8q + 7 (lane 8q + r holds its row r),
// so the chunk states are read in parallel instead of one chunk after another.
constexpr int kFinPerWarp = kWarp / kChunk;
template <int NT>
__device__ void finalize_chunks(const FfnLaunch& a, GateUpShared<NT>& sh, volatile ChunkState<NT>* tab, int c0,
                                int nc, int lane) {
    const int q = lane / kChunk, r = lane % kChunk;
    const bool on = q < nc;
    volatile ChunkState<NT>& s = tab[c0 + (on ? q : 0)];
    const int e = s.e;
    const int chunk = s.chunk;
    const int ntok = sh.es.ntok[e];
    const unsigned gm = s.gmask;
    const int j = on ? s.jr[r] : -1;
    const bool up_row = on && ((gm >> r) & 1u);
    float g[NT], u[NT];
#pragma unroll
    for (int k = 0; k < NT; ++k) {
        g[k] = on ? s.g[r][k] : 0.0f;
        u[k] = up_row ? s.u[r][k] : 0.0f;
    }
    unsigned ub = 0u;
    uint8_t* gb = a.gbits + (size_t)e * a.bits_expert_stride + chunk;
    uint8_t* bb = a.bbits + (size_t)e * a.bits_expert_stride + chunk;
    bool both[NT];
#pragma unroll
    for (int k = 0; k < NT; ++k) {
        const bool gk = j >= 0 && g[k] > 0.0f;
        both[k] = gk && up_row && u[k] > 0.0f;
        // this lane's group's byte of the warp-wide ballots
        const unsigned gbyte = (__ballot_sync(0xffffffffu, gk) >> (kChunk * q)) & 0xffu;
        const unsigned bbyte = (__ballot_sync(0xffffffffu, both[k]) >> (kChunk * q)) & 0xffu;
        if (k < ntok) {
            ub |= bbyte;
            if (on && r == 0) {
                const size_t tb = (size_t)(a.bits_tok_base + k) * a.nbytes;
                gb[tb] = (uint8_t)gbyte;
                bb[tb] = (uint8_t)bbyte;
            }
        }
    }
    if (on && r == 0) {
        a.ubits[(size_t)e * a.nbytes + chunk] = (uint8_t)ub;
        a.ugbits[(size_t)e * a.nbytes + chunk] = (uint8_t)gm;
    }
    const bool b_row = on && ((ub >> r) & 1u);
    // The down projection will gather these W_down rows: pull them into L2
    // now, while HBM is streaming anyway.
    if (b_row)
        prefetch_l2_bulk(static_cast<const unsigned char*>(a.ex[e].wd) + (size_t)j * a.row_bytes,
                         (unsigned)a.row_bytes);
    // c by batch slot: the pass-local token (single FFN) or the global token
    // (MoE, 0 for tokens not routed to this expert)
    if (b_row) {
        float* cv = a.cval + ((size_t)e * kMaxPass) * a.cval_tok_stride + (size_t)chunk * kChunk + r;
        float val[NT];
#pragma unroll
        for (int k = 0; k < NT; ++k) val[k] = (k < ntok && both[k]) ? sh.es.w[e][k] * (g[k] * u[k]) : 0.0f;
        if (a.route == nullptr) {
#pragma unroll
            for (int k = 0; k < NT; ++k)
                if (k < ntok) cv[(size_t)k * a.cval_tok_stride] = val[k];
        } else {
            for (int t = 0; t < a.batch; ++t) {
                float v = 0.0f;
#pragma unroll
                for (int k = 0; k < NT; ++k)
                    if (k < ntok && sh.es.tok[e][k] == t) v = val[k];
                cv[(size_t)t * a.cval_tok_stride] = v;
            }
        }
    }
    if constexpr (NT <= kAccMaxTokens) {
        const int ql = s.q;
        if (on && ql < kMaxLocal) {
            if (r == 0) sh.pd.ub[ql] = (uint8_t)ub;
#pragma unroll
            for (int t = 0; t < kAccMaxTokens; ++t) {
                float v = 0.0f;
#pragma unroll
                for (int k = 0; k < NT; ++k) {
                    const int slot_of_k = a.route ? sh.es.tok[e][k] : k;
                    if (k < ntok && both[k] && slot_of_k == t) v = sh.es.w[e][k] * (g[k] * u[k]);
                }
                sh.pd.c[ql][r][t] = v;
            }
        }
    }
    __syncwarp();
}
template <int NT>
__device__ void finalize_chunk(const FfnLaunch& a, GateUpShared<NT>& sh, int cw, int lane) {
    finalize_chunks<NT>(a, sh, sh.cs, cw, 1, lane);
    __threadfence_block();
    if (lane == 0) mbar_arrive(&sh.chunk_free[cw]);
}

// This CTA's share of the down projection (Eq. 1 over the non-zero
// activations of Eq. 2), once every chunk of the CTA is finalized: for each
// batch slot t,
//     partial[cta][t][:] = sum over the CTA's both-active rows j, in local
//                          chunk order and row order, of c_{t,j} W_down[j,:].
// Consumer warp 0 lists the rows (their W_down address and c values) in
// shared memory, kRoundCap per round; every consumer warp then reads its
// column blocks of those rows straight from L2 (the finalizer prefetched
// them), all blocks of a group of rows in flight at once, and accumulates in
// registers. A round after the first adds onto the stored partial, so the
// order stays fixed and the result is bitwise reproducible.
constexpr int kPartialLoads = 16;  // 16-byte W_down loads a lane has in flight in the down partial

template <typename T, int NT, int NB>
__device__ __forceinline__ void partial_blocks(const FfnLaunch& a, GateUpShared<NT>& sh, int n, int blk0,
                                               int bstride, float* pbase, bool accumulate, int lane) {
    constexpr int VEC = Vec<T>::N;
    constexpr int BLK = kWarp * VEC;
    constexpr int AT = NT;      // batch slots held (NT <= kAccMaxTokens)
    constexpr int U = kPartialLoads / NB;  // rows per group: kPartialLoads loads in flight per lane
    const int d = a.d;
    const int n_slots = a.route ? a.batch : a.nt;
    int col[NB];
    bool valid[NB];
    float acc[NB][AT][VEC];
#pragma unroll
    for (int b = 0; b < NB; ++b) {
        col[b] = (blk0 + b * bstride) * BLK + lane * VEC;
        valid[b] = col[b] < d;
#pragma unroll
        for (int t = 0; t < AT; ++t)
#pragma unroll
            for (int v = 0; v < VEC; ++v)
                acc[b][t][v] = (accumulate && valid[b] && t < n_slots) ? pbase[(size_t)t * d + col[b] + v] : 0.0f;
    }
    for (int g = 0; g < n; g += U) {
        uint4 w[U][NB];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const T* row = g + u < n ? reinterpret_cast<const T*>(sh.pd.rowp[g + u]) : nullptr;
#pragma unroll
            for (int b = 0; b < NB; ++b)
                w[u][b] = (row != nullptr && valid[b]) ? ld_stream(row + col[b]) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            if (g + u < n) {
                float c[AT];
#pragma unroll
                for (int t = 0; t < AT; ++t) c[t] = sh.pd.cs[g + u][t];
#pragma unroll
                for (int b = 0; b < NB; ++b) {
                    float f[VEC];
                    Vec<T>::unpack(w[u][b], f);
#pragma unroll
                    for (int t = 0; t < AT; ++t)
                        if (t < n_slots)
#pragma unroll
                            for (int v = 0; v < VEC; ++v) acc[b][t][v] = fmaf(c[t], f[v], acc[b][t][v]);
                }
            }
        }
    }
#pragma unroll
    for (int b = 0; b < NB; ++b)
        if (valid[b]) {
#pragma unroll
            for (int t = 0; t < AT; ++t)
                if (t < n_slots) {
                    float4* o = reinterpret_cast<float4*>(pbase + (size_t)t * d + col[b]);
#pragma unroll
                    for (int v = 0; v < VEC; v += 4)
                        o[v / 4] = make_float4(acc[b][t][v], acc[b][t][v + 1], acc[b][t][v + 2], acc[b][t][v + 3]);
                }
        }
}

// INT4 rows: in a 512-column block, lanes 2q and 2q+1 share group q (32
// columns, 16 code bytes, one scale); lane parity p reads code words 2p and
// 2p+1, which hold the group's columns 8s + 4p + {0..3} (s = 0..3). Each lane
// so covers 16 columns, for U rows at a time.
__device__ __forceinline__ uint2 ld_nc_u2(const void* p) {
    uint2 v;
    asm volatile("ld.global.nc.L1::no_allocate.v2.u32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "l"(p));
    return v;
}
__device__ __forceinline__ float ld_nc_half(const void* p) {
    unsigned short v;
    asm volatile("ld.global.nc.u16 %0, [%1];" : "=h"(v) : "l"(p));
    return __half2float(__ushort_as_half(v));
}

template <int NT>
__device__ __forceinline__ void partial_blocks_q4(const FfnLaunch& a, GateUpShared<NT>& sh, int n, int blk,
                                                  float* pbase, bool accumulate, int lane) {
    constexpr int AT = NT;
    constexpr int U = 8;
    const int d = a.d;
    const int n_slots = a.route ? a.batch : a.nt;
    const int grp = blk * 16 + lane / 2;
    const int p = lane % 2;
    const int col0 = grp * 32 + 4 * p;  // columns col0 + 8s + {0..3}
    const bool valid = grp * 32 < d;
    // acc[t][4s + c] is column col0 + 8s + c
    float acc[AT][16];
#pragma unroll
    for (int t = 0; t < AT; ++t)
#pragma unroll
        for (int v = 0; v < 16; ++v)
            acc[t][v] = (accumulate && valid && t < n_slots) ? pbase[(size_t)t * d + col0 + 8 * (v / 4) + v % 4] : 0.0f;
    for (int g = 0; g < n; g += U) {
        uint2 cw[U];
        float sc[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const unsigned char* row = g + u < n ? static_cast<const unsigned char*>(sh.pd.rowp[g + u]) : nullptr;
            cw[u] = make_uint2(0x88888888u, 0x88888888u);  // codes of weight 0
            sc[u] = 0.0f;
            if (row != nullptr && valid) {
                cw[u] = ld_nc_u2(row + grp * 16 + 8 * p);
                sc[u] = ld_nc_half(row + d / 2 + grp * 2);
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            if (g + u < n) {
                float c[AT];
#pragma unroll
                for (int t = 0; t < AT; ++t) c[t] = sh.pd.cs[g + u][t] * sc[u];
#pragma unroll
                for (int v = 0; v < 16; ++v) {
                    // column 8s + 2tw + h of the lane's pair: word tw, nibble s + 4h
                    const int s4 = v / 4, tw = (v % 4) / 2, h = v % 2;
                    const uint32_t word = tw ? cw[u].y : cw[u].x;
                    // 2^23 + code as a float, minus 2^23 + 8: code - 8, exact
                    const float q = __uint_as_float(0x4B000000u | ((word >> (4 * s4 + 16 * h)) & 15u)) - 8388616.0f;
#pragma unroll
                    for (int t = 0; t < AT; ++t)
                        if (t < n_slots) acc[t][v] = fmaf(c[t], q, acc[t][v]);
                }
            }
        }
    }
    if (valid) {
#pragma unroll
        for (int t = 0; t < AT; ++t)
            if (t < n_slots) {
#pragma unroll
                for (int s4 = 0; s4 < 4; ++s4)
                    *reinterpret_cast<float4*>(pbase + (size_t)t * d + col0 + 8 * s4) =
                        make_float4(acc[t][4 * s4], acc[t][4 * s4 + 1], acc[t][4 * s4 + 2], acc[t][4 * s4 + 3]);
            }
    }
}

template <typename T, int NT, bool Q4 = false, int C = GateUpWarps<NT>::C>
__device__ void down_partial(const FfnLaunch& a, GateUpShared<NT>& sh, int i0, int i1, int n_chunks, int cidx,
                             int lane) {
    constexpr int VEC = Vec<T>::N;
    constexpr int BLK = kWarp * VEC;
    constexpr int AT = kAccMaxTokens;
    const int cthreads = C * kWarp;
    const int d = a.d;
    const int n_slots = a.route ? a.batch : a.nt;
    float* pbase = a.partial + (size_t)blockIdx.x * a.partial_slots * d;
    const int nblk = (d + BLK - 1) / BLK;
    const int my_blocks = cidx < nblk ? (nblk - 1 - cidx) / C + 1 : 0;
    int it = i0;
    unsigned round = 0;
    do {
        if (cidx == 0) {
            // the rows of the next items, whole items only, at most kRoundCap
            int n = 0;
            bool full = false;
            while (!full && it < i1) {
                const int item = it + lane;
                const int q = item - i0;
                unsigned bits = 0u;
                int e = 0, chunk = 0;
                if (item < i1) {
                    const int ea = item / n_chunks;
                    chunk = item - ea * n_chunks;
                    e = sh.es.act[ea];
                    bits = q < kMaxLocal ? (unsigned)sh.pd.ub[q]
                                         : (unsigned)*reinterpret_cast<const volatile uint8_t*>(
                                               a.ubits + (size_t)e * a.nbytes + chunk);
                    const int left = a.n_rows - chunk * kChunk;  // rows of the row space in this chunk
                    if (left < kChunk) bits &= (1u << (left > 0 ? left : 0)) - 1u;
                }
                const int cnt = __popc(bits);
                int incl = cnt;
#pragma unroll
                for (int o = 1; o < kWarp; o <<= 1) {
                    const int v = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += v;
                }
                // the items that fit are a prefix of the lanes
                const bool fits = item < i1 && n + incl <= kRoundCap;
                const unsigned take = __ballot_sync(0xffffffffu, fits);
                const int n_take = __popc(take);
                if (fits) {
                    int pos = n + incl - cnt;
                    for (unsigned b = bits; b; b &= b - 1u) {
                        const int r = __ffs(b) - 1;
                        const int p = chunk * kChunk + r;
                        int j = a.rows ? a.rows[p] : p;
                        if ((unsigned)j >= (unsigned)a.m) j = 0;  // only after a failed wait: stay in bounds
                        sh.pd.rowp[pos] = static_cast<const unsigned char*>(a.ex[e].wd) + (size_t)j * a.row_bytes;
#pragma unroll
                        for (int t = 0; t < AT; ++t)
                            sh.pd.cs[pos][t] =
                                q < kMaxLocal ? sh.pd.c[q][r][t]
                                              : (t < n_slots ? a.cval[((size_t)e * kMaxPass + t) * a.cval_tok_stride + p]
                                                             : 0.0f);
                        ++pos;
                    }
                }
                if (n_take > 0) n += __shfl_sync(0xffffffffu, incl, n_take - 1);
                it += n_take;
                full = n_take < kWarp && it < i1;  // the next item did not fit
            }
            if (lane == 0) {
                sh.pd.n_rows = n;
                sh.pd.next_item = it;
            }
        }
        named_bar_sync(1, cthreads);
        const int n = sh.pd.n_rows;
        const int next = sh.pd.next_item;
        if constexpr (Q4) {
            for (int b = cidx; b < (d + 511) / 512; b += C) partial_blocks_q4<NT>(a, sh, n, b, pbase, round > 0, lane);
        } else if (my_blocks == 2) {
            partial_blocks<T, NT, 2>(a, sh, n, cidx, C, pbase, round > 0, lane);
        } else {
            for (int b = 0; b < my_blocks; ++b)
                partial_blocks<T, NT, 1>(a, sh, n, cidx + b * C, C, pbase, round > 0, lane);
        }
        it = next;
        ++round;
        named_bar_sync(1, cthreads);  // the list is rebuilt next round
    } while (it < i1);
}

// Single-thread wait that records a timeout in the status word.
__device__ __forceinline__ bool wait_or_flag(uint64_t* bar, unsigned parity, unsigned* status) {
    if (mbar_wait(bar, parity)) return true;
    atomicOr(status, kStatusTimeout);
    return false;
}

// The producer: one thread (lane 0 of warp 0) issuing row copies in task order.
template <typename T, int NT>
__device__ void produce(const FfnLaunch& a, GateUpShared<NT>& sh, unsigned char* ring,
                        const GateUpCfg& cfg, int i0, int i1, int n_chunks) {
    const unsigned S = (unsigned)cfg.slots;
    const unsigned row_bytes = (unsigned)(a.d * sizeof(T));
    const size_t row_elems = (size_t)a.d;
    unsigned slot = 0, phase = 0, issued = 0;  // next slot, its use parity, tasks issued
    bool ok = true;

    // One task: row j of matrix w, for row r of the chunk in window slot cw.
    auto emit = [&](int kind, int cw, int r, int j, const T* w) {
        if (!wait_or_flag(&sh.empty[slot], phase ^ 1u, a.status)) {
            ok = false;
            return;
        }
        sh.task[slot] = Task{r, cw, kind, 0};
        if (kind == kTaskEnd) {
            mbar_arrive(&sh.full[slot]);
        } else {
            mbar_arrive_expect_tx(&sh.full[slot], row_bytes);
            tma_load_1d(ring + (size_t)slot * cfg.slot_bytes, w + (size_t)debug_row(j, a.m, a.status) * row_elems, row_bytes,
                        &sh.full[slot]);
        }
        ++issued;
        if (++slot == S) {
            slot = 0;
            phase ^= 1u;
        }
    };

    const int n_local = i1 - i0;
    int jr_hist[kWindow][kChunk];  // the producer's own copy of each window chunk's rows
    for (int c = 0; ok && c < n_local + kLookahead; ++c) {
        if (c < n_local) {
            const int cw = c % kWindow;
            ok = wait_or_flag(&sh.chunk_free[cw], ((unsigned)(c / kWindow) & 1u) ^ 1u, a.status);
            if (!ok) break;
            const int item = i0 + c;
            const int ea = item / n_chunks;
            const int chunk = item - ea * n_chunks;
            const int e = sh.es.act[ea];
            volatile ChunkState<NT>& s = sh.cs[cw];
            int* jr = jr_hist[cw];
            int n_gate = 0;
#pragma unroll
            for (int r = 0; r < kChunk; ++r) {
                const int p = chunk * kChunk + r;
                int j = -1;
                if (p < a.n_rows) {
                    if (a.rows != nullptr) {
                        const int jj = a.rows[p];
                        if ((unsigned)jj < (unsigned)a.m && (p == 0 || a.rows[p - 1] < jj))
                            j = jj;
                        else
                            atomicOr(a.status, kStatusBadIndex);
                    } else {
                        j = p;
                    }
                }
                jr[r] = j;
                s.jr[r] = j;
                n_gate += j >= 0;
            }
            s.e = e;
            s.chunk = chunk;
            s.q = c;
            s.n_gate = n_gate;
            s.gate_cnt = 0;
            s.up_cnt = 0;
            s.gmask = 0u;
            if (n_gate == 0) {
                // nothing to compute: the chunk's bytes are zero, no c values
                const int ntok = sh.es.ntok[e];
                for (int k = 0; k < ntok; ++k) {
                    const size_t tb = (size_t)(a.bits_tok_base + k) * a.nbytes;
                    a.gbits[(size_t)e * a.bits_expert_stride + chunk + tb] = 0;
                    a.bbits[(size_t)e * a.bits_expert_stride + chunk + tb] = 0;
                }
                a.ubits[(size_t)e * a.nbytes + chunk] = 0;
                a.ugbits[(size_t)e * a.nbytes + chunk] = 0;
                if constexpr (NT <= kAccMaxTokens) {
                    if (c < kMaxLocal) sh.pd.ub[c] = 0;
                }
                mbar_arrive(&sh.chunk_free[cw]);
                mbar_arrive(&sh.gate_ready[cw]);
            } else {
                const T* wg = static_cast<const T*>(a.ex[e].wg);
                for (int r = 0; r < kChunk && ok; ++r)
                    if (jr[r] >= 0) emit(kTaskGate, cw, r, jr[r], wg);
            }
        }
        if (ok && c >= kLookahead) {
            const int cp = c - kLookahead;
            const int cw = cp % kWindow;
            ok = wait_or_flag(&sh.gate_ready[cw], (unsigned)(cp / kWindow) & 1u, a.status);
            if (!ok) break;
            volatile ChunkState<NT>& s = sh.cs[cw];
            const unsigned gm = s.gmask;
            const T* wu = static_cast<const T*>(a.ex[s.e].wu);
            const int* jr = jr_hist[cw];
            for (unsigned m = gm; m && ok; m &= m - 1u) {
                const int r = __ffs(m) - 1;
                emit(kTaskUp, cw, r, jr[r], wu);
            }
        }
    }
    for (int w = 0; w < GateUpWarps<NT>::C && ok; ++w) emit(kTaskEnd, 0, 0, 0, nullptr);
    // copies in flight must land before the CTA exits: wait on the last use of every slot
    for (unsigned q = 0; q < S && q < issued; ++q) {
        slot = slot == 0 ? S - 1 : slot - 1;
        if (slot == S - 1) phase ^= 1u;
        if (!wait_or_flag(&sh.full[slot], phase, a.status)) break;
    }
}

template <typename T, int NT>
__device__ void consume(const FfnLaunch& a, GateUpShared<NT>& sh, const unsigned char* ring,
                        const float* xs, const GateUpCfg& cfg, int cidx, int lane) {
    const unsigned S = (unsigned)cfg.slots;
    constexpr int C = GateUpWarps<NT>::C;
    // consumer cidx owns slots cidx, cidx + C, ... (S is a multiple of C)
    unsigned slot = (unsigned)cidx, phase = 0;
    if (a.test_stall && cidx == 0) {
        // the failure-detection test: a wait that can only run out
        if (!warp_wait(&sh.never, 0u, lane, a.status)) return;
    }
    for (;;) {
        if (!warp_wait(&sh.full[slot], phase, lane, a.status)) return;
        const Task tk = sh.task[slot];
        if (tk.kind == kTaskEnd) return;
        volatile ChunkState<NT>& s = sh.cs[tk.cw];
        const int e = s.e;
        const int ntok = sh.es.ntok[e];
        int xt[NT];
#pragma unroll
        for (int k = 0; k < NT; ++k) xt[k] = k < ntok ? (a.route ? sh.es.tok[e][k] : k) : 0;
        float acc[NT];
        smem_row_dot<T, NT>(ring + (size_t)slot * cfg.slot_bytes, xs, cfg.xs_stride, xt, ntok, a.d, lane,
                            acc);
        __syncwarp();
        if (lane == 0) {
            mbar_arrive(&sh.empty[slot]);
            volatile float* dst = tk.kind == kTaskGate ? s.g[tk.r] : s.u[tk.r];
#pragma unroll
            for (int k = 0; k < NT; ++k) dst[k] = acc[k];
        }
        slot += C;
        if (slot >= S) {
            slot -= S;
            phase ^= 1u;
        }
        __threadfence_block();
        int last = 0;
        if (lane == 0) {
            if (tk.kind == kTaskGate)
                last = atomicAdd((int*)&s.gate_cnt, 1) + 1 == s.n_gate;
            else
                last = atomicAdd((int*)&s.up_cnt, 1) + 1 == __popc(s.gmask);
        }
        last = __shfl_sync(0xffffffffu, last, 0);
        if (!last) continue;
        __threadfence_block();
        if (tk.kind == kTaskGate) {
            // every gate row of the chunk is in: which rows need their W_up row?
            bool ga = false;
            if (lane < kChunk && s.jr[lane] >= 0) {
#pragma unroll
                for (int k = 0; k < NT; ++k) ga |= (k < ntok) && (s.g[lane][k] > 0.0f);
            }
            const unsigned gm = __ballot_sync(0xffffffffu, ga);
            if (lane == 0) s.gmask = gm;
            __syncwarp();
            __threadfence_block();
            if (gm == 0u) finalize_chunk<NT>(a, sh, tk.cw, lane);
            if (lane == 0) mbar_arrive(&sh.gate_ready[tk.cw]);
        } else {
            finalize_chunk<NT>(a, sh, tk.cw, lane);
        }
    }
}

template <typename T, int NT>
__global__ void __launch_bounds__(GateUpWarps<NT>::THREADS, 1) k_gate_up(const FfnLaunch a, const GateUpCfg cfg) {
    __shared__ GateUpShared<NT> sh;
    extern __shared__ __align__(128) unsigned char dyn[];
    float* xs = reinterpret_cast<float*>(dyn);  // [tokens][xs_stride]
    const int n_x = a.route ? a.batch : a.nt;
    unsigned char* ring = dyn + (size_t)n_x * cfg.xs_stride * sizeof(float);

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) {
        for (int s = 0; s < cfg.slots; ++s) {
            mbar_init(&sh.full[s], 1);
            mbar_init(&sh.empty[s], 1);
        }
        for (int w = 0; w < kWindow; ++w) {
            mbar_init(&sh.gate_ready[w], 1);
            mbar_init(&sh.chunk_free[w], 1);
        }
        mbar_init(&sh.never, 1);
        if constexpr (NT <= kAccMaxTokens) {
            for (int q = 0; q < kMaxLocal; ++q) sh.pd.ub[q] = 0;
        }
        mbar_fence_init();
    }
    // Single FFN in detected mode: nothing the producer reads comes from an
    // earlier kernel, so only the consumers wait for it (below).
    const bool early = a.rows == nullptr && a.route == nullptr;
    if (!early) pdl_wait();
    resolve_experts(a, sh.es);  // ends with __syncthreads (barrier init visible)
    pdl_launch_dependents();

    const int n_chunks = (a.n_rows + kChunk - 1) / kChunk;
    const int n_items = sh.es.n_act * n_chunks;
    const int i0 = (int)((long long)n_items * blockIdx.x / gridDim.x);
    const int i1 = (int)((long long)n_items * (blockIdx.x + 1) / gridDim.x);

    if (warp == 0) {
        if (lane == 0) produce<T, NT>(a, sh, ring, cfg, i0, i1, n_chunks);
        return;
    }
    // consumers: activations into shared memory (after the previous kernel)
    if (early) pdl_wait();
    const int ctid = threadIdx.x - kWarp;
    const int cthreads = GateUpWarps<NT>::C * kWarp;
    const int x_tok0 = a.route ? 0 : a.tok0;
    for (int t = 0; t < n_x; ++t) {
        float* xrow = xs + (size_t)t * cfg.xs_stride;
        stage_act_row<T>(a.norm_from_h ? a.h + (size_t)(x_tok0 + t) * a.d : nullptr,
                         static_cast<const T*>(a.x) + (size_t)(x_tok0 + t) * a.d, a.d, ctid, cthreads, sh.red,
                         XsPut<T>{xrow});
    }
    named_bar_sync(1, cthreads);
    consume<T, NT>(a, sh, ring, xs, cfg, warp - 1, lane);
    if constexpr (NT <= kAccMaxTokens) {
        // every chunk is finalized and every ring copy consumed once all
        // consumers are here (no partial buffer: the caller runs the
        // gathered down kernel after a mask instead)
        named_bar_sync(1, cthreads);
        if (a.partial != nullptr) down_partial<T, NT>(a, sh, i0, i1, n_chunks, warp - 1, lane);
    }
}

// ---------------------------------------------------------------------------
// Passes of 4-8 tokens, bf16, d % 256 == 0: tensor-core variant.
//
// At these batch sizes the per-row dot products are a skinny GEMM
// ([tokens x d] x [d x rows]) that CUDA-core FMAs can no longer hide behind
// HBM. Tasks become groups of up to 8 rows of one chunk (its gate rows, or its
// gate-active up rows), two groups in flight in a ring of 16 padded row slots.
// All consumer warps work on each group, warp w over the w-th K slice, with
// mma.sync m16n8k16 (A = the activations, 8 token rows plus 8 zero rows;
// B = the 8 weight rows; fp32 accumulation); the slices are added in warp
// order, so results do not depend on timing. Rows are padded by 16 bytes in
// shared memory so ldmatrix reads are free of bank conflicts.
// ---------------------------------------------------------------------------
constexpr int kMmaGroups = 2;    // groups in flight
constexpr int kMmaRowPad = 16;   // bytes after every row in shared memory
constexpr int kMmaDAlign = 256;  // d must be a multiple (even K-step count per warp)

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
// d += A * B for one m16n8k16 step; A rows 8-15 are zero (no token there).
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a2, uint32_t b0, uint32_t b1) {
    const uint32_t z = 0u;
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(z), "r"(a2), "r"(z), "r"(b0), "r"(b1));
}

struct MmaCfg {
    int x_stride;   // bytes per activation row in shared memory (d * 2 + kMmaRowPad)
    int w_stride;   // bytes per weight row in shared memory (row bytes + kMmaRowPad)
    int groups;     // row groups in flight (kMmaGroups bf16, more for the smaller INT4 rows)
    int lookahead;  // gate groups issued ahead of their chunk's up group
    int end_tasks;  // end groups to emit: 1 (all consumers read each group) or one per consumer
};

// The producer of the tensor-core variant: groups in task order (gate rows of
// chunk c, then the up rows of chunk c-1), one expect-tx barrier per group.
template <int NT>
__device__ void produce_mma(const FfnLaunch& a, GateUpShared<NT>& sh, unsigned char* ring, const MmaCfg& mc,
                            int i0, int i1, int n_chunks) {
    const unsigned row_bytes = (unsigned)a.row_bytes;
    const unsigned G = (unsigned)mc.groups;
    unsigned grp = 0;
    bool ok = true;
    auto emit = [&](int kind, int cw, const int* jr, unsigned mask, const unsigned char* w) {
        const unsigned g = grp % G;
        const unsigned ph = (grp / G) & 1u;
        if (!wait_or_flag(&sh.empty[g], ph ^ 1u, a.status)) {
            ok = false;
            return;
        }
        sh.task[g] = Task{(int)mask, cw, kind, 0};
        if (kind == kTaskEnd) {
            mbar_arrive(&sh.full[g]);
        } else {
            mbar_arrive_expect_tx(&sh.full[g], (unsigned)__popc(mask) * row_bytes);
            for (unsigned m = mask; m; m &= m - 1u) {
                const int r = __ffs(m) - 1;
                tma_load_1d(ring + ((size_t)g * kChunk + r) * mc.w_stride,
                            w + (size_t)debug_row(jr[r], a.m, a.status) * a.row_bytes, row_bytes,
                            &sh.full[g]);
            }
        }
        ++grp;
    };
    const int n_local = i1 - i0;
    const int L = mc.lookahead;  // gate groups ahead of their up group
    int jr_hist[kWindow][kChunk];
    for (int c = 0; ok && c < n_local + L; ++c) {
        if (c < n_local) {
            const int cw = c % kWindow;
            ok = wait_or_flag(&sh.chunk_free[cw], ((unsigned)(c / kWindow) & 1u) ^ 1u, a.status);
            if (!ok) break;
            const int item = i0 + c;
            const int ea = item / n_chunks;
            const int chunk = item - ea * n_chunks;
            const int e = sh.es.act[ea];
            volatile ChunkState<NT>& s = sh.cs[cw];
            int* jr = jr_hist[cw];
            unsigned mask = 0u;
#pragma unroll
            for (int r = 0; r < kChunk; ++r) {
                const int p = chunk * kChunk + r;
                int j = -1;
                if (p < a.n_rows) {
                    if (a.rows != nullptr) {
                        const int jj = a.rows[p];
                        if ((unsigned)jj < (unsigned)a.m && (p == 0 || a.rows[p - 1] < jj))
                            j = jj;
                        else
                            atomicOr(a.status, kStatusBadIndex);
                    } else {
                        j = p;
                    }
                }
                jr[r] = j;
                s.jr[r] = j;
                if (j >= 0) mask |= 1u << r;
            }
            s.e = e;
            s.chunk = chunk;
            s.q = c;
            s.n_gate = __popc(mask);
            s.gate_cnt = 0;
            s.up_cnt = 0;
            s.gmask = 0u;
            if (mask == 0u) {
                const int ntok = sh.es.ntok[e];
                for (int k = 0; k < ntok; ++k) {
                    const size_t tb = (size_t)(a.bits_tok_base + k) * a.nbytes;
                    a.gbits[(size_t)e * a.bits_expert_stride + chunk + tb] = 0;
                    a.bbits[(size_t)e * a.bits_expert_stride + chunk + tb] = 0;
                }
                a.ubits[(size_t)e * a.nbytes + chunk] = 0;
                a.ugbits[(size_t)e * a.nbytes + chunk] = 0;
                mbar_arrive(&sh.chunk_free[cw]);
                mbar_arrive(&sh.gate_ready[cw]);
            } else {
                emit(kTaskGate, cw, jr, mask, static_cast<const unsigned char*>(a.ex[e].wg));
            }
        }
        if (ok && c >= L) {
            const int cp = c - L;
            const int cw = cp % kWindow;
            ok = wait_or_flag(&sh.gate_ready[cw], (unsigned)(cp / kWindow) & 1u, a.status);
            if (!ok) break;
            volatile ChunkState<NT>& s = sh.cs[cw];
            const unsigned gm = s.gmask;
            if (gm) emit(kTaskUp, cw, jr_hist[cw], gm, static_cast<const unsigned char*>(a.ex[s.e].wu));
        }
    }
    for (int q = 0; q < mc.end_tasks && ok; ++q) emit(kTaskEnd, 0, nullptr, 0u, nullptr);
    // copies in flight must land before the CTA exits
    for (unsigned q = 0; q < G && q < grp; ++q) {
        const unsigned gi = grp - 1 - q;
        if (!wait_or_flag(&sh.full[gi % G], (gi / G) & 1u, a.status)) break;
    }
}

// The consumers of the tensor-core variant (C warps, all on every group).

template <int NT>
__device__ void consume_mma(const FfnLaunch& a, GateUpShared<NT>& sh, const unsigned char* ring,
                            const unsigned char* xb, float* red, const MmaCfg& mc, int cidx, int lane) {
    constexpr int C = GateUpWarps<NT>::C;
    const int cthreads = C * kWarp;
    const int n_ks = a.d / 16;          // K steps of 16
    const int per = n_ks / C;           // even: d % kMmaDAlign == 0
    const int ks0 = cidx * per;
    const uint32_t x_addr = smem_u32(xb) + (lane % 8) * mc.x_stride + (lane / 8) * 16;
    const unsigned G = (unsigned)mc.groups;
    // All consumer warps meet at named barriers inside every group, so they
    // must agree on whether to go on: one thread waits, the outcome is shared.
    if (cidx == 0 && lane == 0) {
        int ok = 1;
        if (a.test_stall) {
            // the failure-detection test: a wait that can only run out
            ok = mbar_wait(&sh.never, 0u) ? 1 : 0;
            if (!ok) atomicOr(a.status, kStatusTimeout);
        }
        sh.mma_ok = ok;
    }
    for (unsigned grp = 0;; ++grp) {
        const unsigned g = grp % G;
        const unsigned parity = (grp / G) & 1u;
        if (cidx == 0 && lane == 0 && sh.mma_ok) {
            const bool ok = mbar_wait(&sh.full[g], parity);
            if (!ok) atomicOr(a.status, kStatusTimeout);
            sh.mma_ok = ok ? 1 : 0;
        }
        named_bar_sync(1, cthreads);
        if (!sh.mma_ok) return;
        // the phase is complete: every thread's own (immediate) wait makes the copies visible to it
        if (!warp_wait(&sh.full[g], parity, lane, a.status)) return;
        const Task tk = sh.task[g];
        if (tk.kind == kTaskEnd) return;
        float acc0[4] = {0.0f, 0.0f, 0.0f, 0.0f}, acc1[4] = {0.0f, 0.0f, 0.0f, 0.0f};
        {
            const uint32_t w_addr = smem_u32(ring) + (g * kChunk + lane % 8) * mc.w_stride + (lane / 8) * 16;
            for (int ks = ks0; ks < ks0 + per; ks += 2) {
                uint32_t a0, a2, a0n, a2n, b0, b1, b0n, b1n;
                ldsm_x4(x_addr + ks * 32, a0, a2, a0n, a2n);
                ldsm_x4(w_addr + ks * 32, b0, b1, b0n, b1n);
                mma_bf16_16816(acc0, a0, a2, b0, b1);
                mma_bf16_16816(acc1, a0n, a2n, b0n, b1n);
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh.empty[g]);
        // D rows = tokens (lane / 4), columns = rows of the group (2 * (lane % 4) + {0, 1})
        float* rd = red + ((size_t)g * C + cidx) * 64;
        const int tok = lane / 4, col = 2 * (lane % 4);
        rd[tok * 8 + col] = acc0[0] + acc1[0];
        rd[tok * 8 + col + 1] = acc0[1] + acc1[1];
        named_bar_sync(1, cthreads);
        if (cidx < 2) {
            // add the K slices in warp order: 64 (token, row) values
            const int i = cidx * 32 + lane;
            const int t = i / 8, r = i % 8;
            float v = 0.0f;
            const float* rg = red + (size_t)g * C * 64;
#pragma unroll
            for (int w = 0; w < C; ++w) v += rg[w * 64 + i];
            volatile ChunkState<NT>& s = sh.cs[tk.cw];
            const int e = s.e;
            const int ntok = sh.es.ntok[e];
            if ((tk.r >> r) & 1) {
                // token t of the staged activations -> the chunk's batch slot
#pragma unroll
                for (int k = 0; k < NT; ++k) {
                    const int tk_x = a.route ? sh.es.tok[e][k] : k;
                    if (k < ntok && tk_x == t) {
                        if (tk.kind == kTaskGate)
                            s.g[r][k] = v;
                        else
                            s.u[r][k] = v;
                    }
                }
            }
            named_bar_sync(2, 2 * kWarp);
            if (cidx == 0) {
                __threadfence_block();
                if (tk.kind == kTaskGate) {
                    bool ga = false;
                    if (lane < kChunk && s.jr[lane] >= 0) {
#pragma unroll
                        for (int k = 0; k < NT; ++k) ga |= (k < ntok) && (s.g[lane][k] > 0.0f);
                    }
                    const unsigned gm = __ballot_sync(0xffffffffu, ga);
                    if (lane == 0) s.gmask = gm;
                    __syncwarp();
                    __threadfence_block();
                    if (gm == 0u) finalize_chunk<NT>(a, sh, tk.cw, lane);
                    if (lane == 0) mbar_arrive(&sh.gate_ready[tk.cw]);
                } else {
                    finalize_chunk<NT>(a, sh, tk.cw, lane);
                }
            }
        }
    }
}

template <int NT>
__global__ void __launch_bounds__(GateUpWarps<NT>::THREADS, 1) k_gate_up_mma(const FfnLaunch a, const MmaCfg mc) {
    using T = __nv_bfloat16;  // activations (and bf16 weights)
    constexpr int C = GateUpWarps<NT>::C;
    __shared__ GateUpShared<NT> sh;
    extern __shared__ __align__(128) unsigned char dyn[];
    unsigned char* xb = dyn;                                       // [8][x_stride] bf16 activations
    float* red = reinterpret_cast<float*>(dyn + (size_t)kChunk * mc.x_stride);  // [groups][C][64]
    unsigned char* ring = dyn + (size_t)kChunk * mc.x_stride + (size_t)mc.groups * C * 64 * sizeof(float);
    const int n_x = a.route ? a.batch : a.nt;

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) {
        for (int g = 0; g < mc.groups; ++g) {
            mbar_init(&sh.full[g], 1);
            mbar_init(&sh.empty[g], C);
        }
        mbar_init(&sh.never, 1);
        for (int w = 0; w < kWindow; ++w) {
            mbar_init(&sh.gate_ready[w], 1);
            mbar_init(&sh.chunk_free[w], 1);
        }
        mbar_fence_init();
    }
    const bool early = a.rows == nullptr && a.route == nullptr;
    if (!early) pdl_wait();
    resolve_experts(a, sh.es);
    pdl_launch_dependents();

    const int n_chunks = (a.n_rows + kChunk - 1) / kChunk;
    const int n_items = sh.es.n_act * n_chunks;
    const int i0 = (int)((long long)n_items * blockIdx.x / gridDim.x);
    const int i1 = (int)((long long)n_items * (blockIdx.x + 1) / gridDim.x);

    if (warp == 0) {
        if (lane == 0) produce_mma<NT>(a, sh, ring, mc, i0, i1, n_chunks);
        return;
    }
    if (early) pdl_wait();
    const int ctid = threadIdx.x - kWarp;
    const int cthreads = C * kWarp;
    const int x_tok0 = a.route ? 0 : a.tok0;
    // activations as bf16 rows (tokens past the pass are zero)
    for (int t = 0; t < kChunk; ++t) {
        __nv_bfloat16* xrow = reinterpret_cast<__nv_bfloat16*>(xb + (size_t)t * mc.x_stride);
        if (t >= n_x) {
            for (int i = ctid; i < a.d; i += cthreads) xrow[i] = __float2bfloat16_rn(0.0f);
        } else {
            stage_act_row<T>(a.norm_from_h ? a.h + (size_t)(x_tok0 + t) * a.d : nullptr,
                             static_cast<const T*>(a.x) + (size_t)(x_tok0 + t) * a.d, a.d, ctid, cthreads, sh.red,
                             [&](int i, float v) { xrow[i] = __float2bfloat16_rn(v); });
        }
    }
    named_bar_sync(1, cthreads);
    consume_mma<NT>(a, sh, ring, xb, red, mc, warp - 1, lane);
}

// Shared memory of the tensor-core variant: activations, the cross-warp
// sums of every group in flight, and the ring of kMmaGroups bf16 groups.
static size_t mma_smem(int d, MmaCfg* mc) {
    const int row_bytes = d * 2;
    mc->x_stride = d * 2 + kMmaRowPad;
    mc->w_stride = row_bytes + kMmaRowPad;
    auto bytes = [&](int g) {
        return (size_t)kChunk * mc->x_stride + (size_t)g * GateUpWarps<8>::C * 64 * sizeof(float) +
               (size_t)g * kChunk * mc->w_stride;
    };
    const int g = kMmaGroups;
    mc->groups = g;
    mc->lookahead = 1;
    mc->end_tasks = 1;
    return bytes(g);
}

// ---------------------------------------------------------------------------
// INT4 rows, passes of 1-2 tokens. A subtask is up to kQ4Rows rows of one
// chunk (its gate rows, or its gate-active up rows) over the full K,
// computed by one consumer warp from one of its two ring slots.
//
// One m16n8k16 MMA covers the task's 4 rows over all four K-quarters: A row
// g (g < 8) is task row g % 4 over quarter g / 4, A row g + 8 the same row
// over quarter 3 - g / 4; B column n is token n / 4 over quarter (n even:
// (n / 2) % 2, n odd: 2 + (n / 2) % 2). Each lane then holds exactly one
// product of matching quarters, D[g][2t] when g / 4 == t % 2 and
// D[g + 8][2t + 1] otherwise, and the four quarters of a (row, token) sit in
// lanes {l, l ^ 1, l ^ 16, l ^ 17}. Odd quarters walk each pair of groups in
// swapped order, which keeps the lanes' shared-memory words in distinct banks.
// ---------------------------------------------------------------------------
constexpr int kQ4Rows = 4;          // rows per subtask
constexpr int kQ4Consumers = 8;     // consumer warps (10 fit in shared memory but measured no faster)
constexpr int kQ4SlotsPerWarp = 2;  // ring slots per consumer warp
constexpr int kQ4QuarterPad = 16;   // bytes after each K-quarter of an activation row
// bytes of the activations' 32-element group sums (kAccMaxTokens rows)
__host__ __device__ constexpr size_t q4_xsum_bytes(int d) {
    return ((size_t)kAccMaxTokens * (d / 32) * sizeof(float) + 127) / 128 * 128;
}

// bf16x2 A-fragment register of two INT4 codes held at bits 0-3 and 16-19
// of v: (128 + code_lo, 128 + code_hi), exact. 0x4300 is 128.0 in bf16,
// whose last mantissa bit is worth 1.0, so OR-ing a code into it gives
// 128 + code. The dequantized weight is code - 8: a group's dot product with
// these pairs is corrected afterwards by 136 times the group's activation
// sum, one fma per group instead of a subtraction per pair.
__device__ __forceinline__ uint32_t q4_frag(uint32_t v) { return (v & 0x000F000Fu) | 0x43004300u; }
// d += A * B for one m16n8k16 step with all 16 A rows.
__device__ __forceinline__ void mma_bf16_16816_a4(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                                  uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Each chunk's rows are computed in subtasks of up to kQ4Rows rows, and the
// CTA's chunks are taken in rounds of up to kQ4Round: first every gate
// subtask of the round (the rows of each chunk half), shared out one at a
// time to whichever consumer warp asks next; then, once the round's gate
// values are in, every up subtask (a chunk's gate-active rows, four at a
// time), shared out the same way; then the chunks are finalized. The
// subtasks of a phase are independent, so no warp waits on another until
// the phase ends, and the work is balanced to one subtask. A warp copies
// the rows of its next subtask (16-byte cp.async per lane, into the other
// of its two slots) before it computes the current one.
constexpr int kQ4Round = kMaxLocal;  // chunks per round

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

template <int NT, typename Stage>
__device__ void consume_q4w(const FfnLaunch& a, GateUpShared<NT>& sh, unsigned char* ring, const unsigned char* xb,
                            const float* xsum, ChunkState<NT>* tab, const MmaCfg& mc, int i0, int i1, int n_chunks,
                            int cidx, int lane, Stage stage) {
    constexpr int C = kQ4Consumers;
    const int cthreads = C * kWarp;
    const int d = a.d;
    const int nq = d / 128;  // 32-element groups per K-quarter
    const int g = lane / 4, t = lane % 4;
    const int wr = g % 4;                  // subtask row of this lane's A rows
    const int qa = g / 4, qb = 3 - g / 4;  // their K-quarters
    const bool use_d0 = qa == (t & 1);     // which D element holds this lane's product
    const int qu = use_d0 ? qa : qb;       // the quarter of that product
    // A words: word t of each group of the lane's two quarters, for a pair
    // of groups (G, G + 1) at once by ldmatrix: this lane addresses row
    // lane % 8 of matrix lane / 8, i.e. the 16 code bytes of subtask row
    // (lane % 8) % 4 in quarter qa (matrices 0, 2) or qb (1, 3) of group G
    // (matrices 0, 1) or G + 1 (2, 3); odd quarters take the pair in the
    // order (G + 1, G).
    const int lg = lane % 8, lm = lane / 8;
    const int l_q = (lm & 1) ? 3 - lg / 4 : lg / 4;
    const int l_off = l_q * (d / 8) + (((lm >> 1) ^ (l_q & 1)) * 16);
    // B: this lane addresses column n = lane % 8 for ldmatrix; with one
    // token, columns 4-7 repeat token 0 (same addresses, no bank conflict)
    // and their products are not used
    const int n = lane % 8;
    const int n_tok = NT > 1 ? n / 4 : 0;
    // activation sums of the groups of this lane's product (token t / 2)
    const float* xg = xsum + (NT > 1 ? t / 2 : 0) * (d / 32) + qu * nq;
    const int n_q = (n & 1) ? 2 + ((n >> 1) & 1) : ((n >> 1) & 1);
    const uint32_t x_col = smem_u32(xb) + n_tok * mc.x_stride + n_q * (d / 2 + kQ4QuarterPad) + (lane / 8) * 16;
    const uint32_t x_step = 64u;
    const uint32_t x_off0 = (n_q & 1) ? x_step : 0u, x_off1 = x_step - x_off0;
    const unsigned row_bytes = (unsigned)a.row_bytes;
    const int row_chunks = (int)(row_bytes / 16);
    const int n_local = i1 - i0;
    // the failure-detection test: one warp's wait that can only run out
    if (a.test_stall && cidx == 0) warp_wait(&sh.never, 0u, lane, a.status);

    // copy a subtask's rows into this warp's slot `slot` (one commit group)
    auto issue = [&](int kind, int c, unsigned rows, int slot) {
        volatile ChunkState<NT>& s = tab[c];
        const int e = s.e;
        const unsigned char* w = static_cast<const unsigned char*>(kind == kTaskGate ? a.ex[e].wg : a.ex[e].wu);
        unsigned char* dst = ring + (size_t)(2 * cidx + slot) * kQ4Rows * mc.w_stride;
        int i = 0;
        for (unsigned m = rows; m; m &= m - 1u, ++i) {
            const int j = debug_row(s.jr[__ffs(m) - 1], a.m, a.status);
            const unsigned char* src = w + (size_t)j * row_bytes;
            unsigned char* drow = dst + (size_t)i * mc.w_stride;
            for (int k = lane; k < row_chunks; k += kWarp) cp_async16(drow + 16 * k, src + 16 * k);
        }
        cp_async_commit();
    };
    // dot products of the subtask's rows (slot `slot`) with the staged tokens
    auto compute = [&](int kind, int c, unsigned rows, int slot) {
        const unsigned char* sbase = ring + (size_t)(2 * cidx + slot) * kQ4Rows * mc.w_stride;
        const unsigned char* row = sbase + (size_t)wr * mc.w_stride;
        const uint32_t c_addr = smem_u32(sbase + (size_t)(lg % 4) * mc.w_stride + l_off);
        const unsigned char* sp = row + d / 2 + qu * nq * 2;  // binary16 scales of quarter qu
        float v0 = 0.0f, v1 = 0.0f;
#pragma unroll 4
        for (int G = 0; G < nq; G += 2) {
            const float2 sc = __half22float2(*reinterpret_cast<const __half2*>(sp + G * 2));
            const float s0 = (qu & 1) ? sc.y : sc.x;
            const float s1 = (qu & 1) ? sc.x : sc.y;
            const float2 xs = *reinterpret_cast<const float2*>(xg + G);
            const float x0 = (qu & 1) ? xs.y : xs.x;
            const float x1 = (qu & 1) ? xs.x : xs.y;
            uint32_t cw[4];  // (qa, G), (qb, G), (qa, G + 1), (qb, G + 1) in this lane's order
            ldsm_x4(c_addr + G * 16, cw[0], cw[1], cw[2], cw[3]);
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                uint32_t b0, b1, b0n, b1n;
                ldsm_x4(x_col + G * x_step + (h ? x_off1 : x_off0), b0, b1, b0n, b1n);
                const uint32_t ca = cw[2 * h];
                const uint32_t cb = cw[2 * h + 1];
                // element 8s + 2t + {0, 1} of a group is nibble s (+4) of word t;
                // the group's two K-steps go to separate accumulators, so the
                // two MMAs do not wait on each other
                float dg[4] = {0.0f, 0.0f, 0.0f, 0.0f}, dh[4] = {0.0f, 0.0f, 0.0f, 0.0f};
                mma_bf16_16816_a4(dg, q4_frag(ca), q4_frag(cb), q4_frag(ca >> 4), q4_frag(cb >> 4), b0, b1);
                mma_bf16_16816_a4(dh, q4_frag(ca >> 8), q4_frag(cb >> 8), q4_frag(ca >> 12), q4_frag(cb >> 12), b0n,
                                  b1n);
                // sum over the group of (128 + code) x, less 136 times the sum of x
                const float pv = use_d0 ? dg[0] + dh[0] : dg[3] + dh[3];
                if (h == 0)
                    v0 = fmaf(s0, fmaf(-136.0f, x0, pv), v0);
                else
                    v1 = fmaf(s1, fmaf(-136.0f, x1, pv), v1);
            }
        }
        // the four K-quarters of (row wr, token t / 2), in the same order in every lane
        float v = v0 + v1;
        v += __shfl_xor_sync(0xffffffffu, v, 1);
        v += __shfl_xor_sync(0xffffffffu, v, 16);
        volatile ChunkState<NT>& s = tab[c];
        const int e = s.e;
        const int ntok = sh.es.ntok[e];
        if (g < kQ4Rows && (t & 1) == 0 && wr < __popc(rows)) {
            const int r = __fns(rows, 0, wr + 1);  // chunk row of subtask row wr
            const int tok = t / 2;
#pragma unroll
            for (int k = 0; k < NT; ++k) {
                const int tk_x = a.route ? sh.es.tok[e][k] : k;
                if (k < ntok && tk_x == tok) {
                    if (kind == kTaskGate)
                        s.g[r][k] = v;
                    else
                        s.u[r][k] = v;
                }
            }
        }
        __syncwarp();
    };

    // the round's chunks: rows, expert, local index (warp w sets up chunks w, w + C, ...)
    auto setup = [&](int base, int nr) {
        for (int c = cidx; c < nr; c += C) {
            const int item = i0 + base + c;
            const int ea = item / n_chunks;
            const int chunk = item - ea * n_chunks;
            const int e = sh.es.act[ea];
            volatile ChunkState<NT>& s = tab[c];
            int j = -1;
            const int p = chunk * kChunk + lane;
            if (lane < kChunk && p < a.n_rows) {
                if (a.rows != nullptr) {
                    const int jj = a.rows[p];
                    if ((unsigned)jj < (unsigned)a.m && (p == 0 || a.rows[p - 1] < jj))
                        j = jj;
                    else
                        atomicOr(a.status, kStatusBadIndex);
                } else {
                    j = p;
                }
            }
            if (lane < kChunk) s.jr[lane] = j;
            const unsigned mask = __ballot_sync(0xffffffffu, j >= 0);
            if (lane == 0) {
                s.e = e;
                s.chunk = chunk;
                s.q = base + c;
                s.n_gate = (int)mask;  // the chunk's row mask
                s.gmask = 0u;
            }
        }
        if (cidx == 0 && lane == 0) {
            sh.q4_ctr[0] = 0;
            sh.q4_ctr[1] = 0;
        }
    };
    // the next subtask of a phase: chunk c, rows `rows`; false when none is left
    auto claim = [&](int phase, int n_sub, int& c, unsigned& rows) -> bool {
        for (;;) {
            int q = 0;
            if (lane == 0) q = atomicAdd(&sh.q4_ctr[phase], 1);
            q = __shfl_sync(0xffffffffu, q, 0);
            if (q >= n_sub) return false;
            if (phase == 0) {
                c = q >> 1;  // gate rows of chunk half q % 2
                rows = (unsigned)tab[c].n_gate & (0xFu << (4 * (q & 1)));
                if (rows == 0u) continue;
            } else {
                const unsigned ent = sh.q4_up[q];
                c = (int)(ent >> 8);
                rows = ent & 0xFFu;
            }
            return true;
        }
    };
    // The weights do not depend on the activations: each warp's first gate
    // rows are set going while the activations are staged, just after the
    // activation loads are issued (so those loads do not queue behind the
    // row copies).
    int c_first = 0;
    unsigned r_first = 0u;
    setup(0, min(kQ4Round, n_local));
    named_bar_sync(1, cthreads);
    bool have_first = false;
    stage([&]() {
        have_first = claim(0, 2 * min(kQ4Round, n_local), c_first, r_first);
        if (have_first) issue(kTaskGate, c_first, r_first, 0);
    });

    for (int base = 0; base < n_local; base += kQ4Round) {
        const int nr = min(kQ4Round, n_local - base);
        if (base > 0) {
            setup(base, nr);
            named_bar_sync(1, cthreads);
        }
        for (int phase = 0; phase < 2; ++phase) {
            const int kind = phase == 0 ? kTaskGate : kTaskUp;
            const int n_sub = phase == 0 ? 2 * nr : sh.q4_ctr[2];
            int c_cur = 0, c_nxt = 0;
            unsigned r_cur = 0u, r_nxt = 0u;
            bool have;
            int slot = 0;
            if (base == 0 && phase == 0) {
                have = have_first;
                c_cur = c_first;
                r_cur = r_first;
            } else {
                have = claim(phase, n_sub, c_cur, r_cur);
                if (have) issue(kind, c_cur, r_cur, slot);
            }
            while (have) {
                const bool have_nxt = claim(phase, n_sub, c_nxt, r_nxt);
                if (have_nxt) {
                    issue(kind, c_nxt, r_nxt, slot ^ 1);
                    cp_async_wait<1>();
                } else {
                    cp_async_wait<0>();
                }
                __syncwarp();  // every lane's copies of the current subtask have landed
                compute(kind, c_cur, r_cur, slot);
                c_cur = c_nxt;
                r_cur = r_nxt;
                have = have_nxt;
                slot ^= 1;
            }
            named_bar_sync(1, cthreads);
            if (phase == 0 && cidx == 0) {
                // gate-active rows of each chunk (lane c), and the up subtasks:
                // the first four of them, then the rest
                unsigned gm = 0u;
                if (lane < nr) {
                    volatile ChunkState<NT>& s = tab[lane];
                    const int ntok = sh.es.ntok[s.e];
                    for (int r = 0; r < kChunk; ++r) {
                        bool ga = false;
                        if (s.jr[r] >= 0) {
#pragma unroll
                            for (int k = 0; k < NT; ++k) ga |= (k < ntok) && (s.g[r][k] > 0.0f);
                        }
                        if (ga) gm |= 1u << r;
                    }
                    s.gmask = gm;
                }
                const int cnt = __popc(gm) > kQ4Rows ? 2 : (gm != 0u ? 1 : 0);
                int incl = cnt;
#pragma unroll
                for (int o = 1; o < kWarp; o <<= 1) {
                    const int v = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += v;
                }
                int pos = incl - cnt;
                unsigned m = gm;
                for (int k = 0; k < cnt; ++k) {
                    unsigned sub = 0u;
                    for (int i = 0; i < kQ4Rows && m != 0u; ++i) {
                        sub |= m & (0u - m);
                        m &= m - 1u;
                    }
                    sh.q4_up[pos++] = ((unsigned)lane << 8) | sub;
                }
                if (lane == kWarp - 1) sh.q4_ctr[2] = incl;
                __syncwarp();
            }
            if (phase == 0) named_bar_sync(1, cthreads);
        }
        for (int c0 = cidx * kFinPerWarp; c0 < nr; c0 += C * kFinPerWarp)
            finalize_chunks<NT>(a, sh, tab, c0, min(kFinPerWarp, nr - c0), lane);
        named_bar_sync(1, cthreads);  // the table is refilled next round
    }
}

template <int NT>
__global__ void __launch_bounds__((kQ4Consumers + 1) * kWarp, 1) k_gate_up_q4w(const FfnLaunch a, const MmaCfg mc) {
    using T = __nv_bfloat16;  // activations
    constexpr int C = kQ4Consumers;
    __shared__ GateUpShared<NT> sh;
    extern __shared__ __align__(128) unsigned char dyn[];
    // [NT][4 quarters][d/4 bf16 + pad] activations, their group sums, the
    // ring, the round's chunks
    unsigned char* xb = dyn;
    const size_t x_bytes = ((size_t)kAccMaxTokens * mc.x_stride + 127) / 128 * 128;
    float* xsum = reinterpret_cast<float*>(dyn + x_bytes);  // [NT][d/32]
    unsigned char* ring = dyn + x_bytes + q4_xsum_bytes(a.d);  // [C][2 slots][kQ4Rows][w_stride]
    ChunkState<NT>* tab = reinterpret_cast<ChunkState<NT>*>(ring + (size_t)mc.groups * kQ4Rows * mc.w_stride);
    const int n_x = a.route ? a.batch : a.nt;

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) {
        mbar_init(&sh.never, 1);
        for (int q = 0; q < kMaxLocal; ++q) sh.pd.ub[q] = 0;
        mbar_fence_init();
    }
    const bool early = a.rows == nullptr && a.route == nullptr;
    if (!early) pdl_wait();
    resolve_experts(a, sh.es);
    pdl_launch_dependents();

    const int n_chunks = (a.n_rows + kChunk - 1) / kChunk;
    const int n_items = sh.es.n_act * n_chunks;
    const int i0 = (int)((long long)n_items * blockIdx.x / gridDim.x);
    const int i1 = (int)((long long)n_items * (blockIdx.x + 1) / gridDim.x);

    if (warp == 0) return;  // the consumer warps copy their own rows
    const int ctid = threadIdx.x - kWarp;
    const int cthreads = C * kWarp;
    const int x_tok0 = a.route ? 0 : a.tok0;
    const int dq = a.d / 4;
    // bf16 index in a row of element i (i < d): K-quarter (i >= dq) + (i >= 2dq) + (i >= 3dq)
    auto xpos = [&](int i) { return i + ((i >= dq) + (i >= 2 * dq) + (i >= 3 * dq)) * (kQ4QuarterPad / 2); };
    // Stage the activations; first_rows() (the first weight-row copies) runs
    // once, right after the first activation loads are issued (issuing them
    // before the dependency wait, as the bf16 kernel does, measured 1% slower
    // here).
    auto stage = [&](auto&& first_rows) {
        if (early) pdl_wait();
        bool started = false;
        auto once = [&]() {
            if (!started) {
                started = true;
                first_rows();
            }
        };
        for (int t = 0; t < NT; ++t) {
            __nv_bfloat16* xrow = reinterpret_cast<__nv_bfloat16*>(xb + (size_t)t * mc.x_stride);
            if (t >= n_x) {
                for (int i = ctid; i < a.d; i += cthreads) xrow[xpos(i)] = __float2bfloat16_rn(0.0f);
            } else {
                stage_act_row<T>(a.norm_from_h ? a.h + (size_t)(x_tok0 + t) * a.d : nullptr,
                                 static_cast<const T*>(a.x) + (size_t)(x_tok0 + t) * a.d, a.d, ctid, cthreads,
                                 sh.red, [&](int i, float v) { xrow[xpos(i)] = __float2bfloat16_rn(v); }, once);
            }
        }
        once();
        named_bar_sync(1, cthreads);
        // each 32-element group's sum of the staged activations, in order
        const int ng = a.d / 32;
        for (int i = ctid; i < NT * ng; i += cthreads) {
            const int t = i / ng;
            const __nv_bfloat16* xr =
                reinterpret_cast<const __nv_bfloat16*>(xb + (size_t)t * mc.x_stride) + xpos((i - t * ng) * 32);
            float sum = 0.0f;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const uint4 v = *reinterpret_cast<const uint4*>(xr + 8 * k);
                const __nv_bfloat162* p = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float2 f = __bfloat1622float2(p[q]);
                    sum += f.x;
                    sum += f.y;
                }
            }
            xsum[i] = sum;
        }
        named_bar_sync(1, cthreads);
    };
    consume_q4w<NT>(a, sh, ring, xb, xsum, tab, mc, i0, i1, n_chunks, warp - 1, lane, stage);
    down_partial<T, NT, true, kQ4Consumers>(a, sh, i0, i1, n_chunks, warp - 1, lane);
}

// Shared memory of the INT4 kernel: activations (kAccMaxTokens rows of four
// padded K-quarters), the ring, and the states of a round's chunks. A slot row's stride is
// 32 bytes past a multiple of 128, which with the swapped order of odd
// quarters puts the 32 lanes' code words in 32 banks.
static size_t q4w_smem(int d, int avail, MmaCfg* mc) {
    const int row_bytes = d / 2 + d / 16;
    mc->x_stride = 4 * (d / 2 + kQ4QuarterPad);
    mc->w_stride = row_bytes + ((32 - row_bytes % 128) % 128 + 128) % 128;
    const size_t x_bytes = ((size_t)kAccMaxTokens * mc->x_stride + 127) / 128 * 128;
    const int C = kQ4Consumers;
    const size_t slot = (size_t)kQ4Rows * mc->w_stride;
    mc->groups = C * kQ4SlotsPerWarp;
    mc->lookahead = 0;
    mc->end_tasks = 0;
    (void)avail;
    return x_bytes + q4_xsum_bytes(d) + (size_t)mc->groups * slot + (size_t)kQ4Round * sizeof(ChunkState<kAccMaxTokens>);
}

// ---------------------------------------------------------------------------
// bf16 rows, passes of 1-2 tokens, without a producer thread. A single
// thread issuing one bulk copy per row sustains only about 3.7 TB/s for
// 8 KB rows, so here every consumer warp copies its own rows (16-byte
// cp.async per lane) into its own ring slots, a few rows ahead of the one it
// computes. The CTA's chunks are taken in rounds, as in the INT4 kernel:
// every gate row of the round is handed to whichever warp asks next, then
// every gate-active up row, then the chunks are finalized.
// ---------------------------------------------------------------------------
constexpr int kRowsMaxAhead = 2;  // rows a warp has in flight besides the one it computes

struct RowsCfg {
    int xs_stride;   // floats per activation row in shared memory
    int slot_bytes;  // bytes per ring slot: one row, rounded up to 128
    int ahead;       // rows in flight per warp besides the current one (1 or 2)
};

template <int N>
__device__ __forceinline__ void cp_async_wait_n(int n) {
    // wait until at most n of this thread's copy groups are pending (n <= N)
    if (n <= 0) {
        cp_async_wait<0>();
    } else if (n == 1 || N == 1) {
        cp_async_wait<1>();
    } else {
        cp_async_wait<2>();
    }
}

template <typename T, int NT, typename Stage>
__device__ void consume_rows(const FfnLaunch& a, GateUpShared<NT>& sh, unsigned char* ring, const float* xs,
                             ChunkState<NT>* tab, unsigned short* ulist, const RowsCfg& rc, int i0, int i1,
                             int n_chunks, int cidx, int lane, Stage stage) {
    constexpr int C = GateUpWarps<NT>::C;
    const int cthreads = C * kWarp;
    const unsigned row_bytes = (unsigned)(a.d * sizeof(T));
    const int row_chunks = (int)(row_bytes / 16);
    const int n_local = i1 - i0;
    const int P = rc.ahead + 1;  // this warp's slots
    // the failure-detection test: one warp's wait that can only run out
    if (a.test_stall && cidx == 0) warp_wait(&sh.never, 0u, lane, a.status);

    auto setup = [&](int base, int nr) {
        for (int c = cidx; c < nr; c += C) {
            const int item = i0 + base + c;
            const int ea = item / n_chunks;
            const int chunk = item - ea * n_chunks;
            const int e = sh.es.act[ea];
            volatile ChunkState<NT>& s = tab[c];
            int j = -1;
            const int p = chunk * kChunk + lane;
            if (lane < kChunk && p < a.n_rows) {
                if (a.rows != nullptr) {
                    const int jj = a.rows[p];
                    if ((unsigned)jj < (unsigned)a.m && (p == 0 || a.rows[p - 1] < jj))
                        j = jj;
                    else
                        atomicOr(a.status, kStatusBadIndex);
                } else {
                    j = p;
                }
            }
            if (lane < kChunk) s.jr[lane] = j;
            const unsigned mask = __ballot_sync(0xffffffffu, j >= 0);
            if (lane == 0) {
                s.e = e;
                s.chunk = chunk;
                s.q = base + c;
                s.n_gate = (int)mask;  // the chunk's row mask
                s.gmask = 0u;
            }
        }
        if (cidx == 0 && lane == 0) {
            sh.q4_ctr[0] = 0;
            sh.q4_ctr[1] = 0;
        }
    };
    // the next row of a phase: chunk c, row r; false when none is left
    auto claim = [&](int phase, int n_sub, int& c, int& r) -> bool {
        for (;;) {
            int q = 0;
            if (lane == 0) q = atomicAdd(&sh.q4_ctr[phase], 1);
            q = __shfl_sync(0xffffffffu, q, 0);
            if (q >= n_sub) return false;
            if (phase == 0) {
                c = q / kChunk;
                r = q % kChunk;
                if ((((unsigned)tab[c].n_gate >> r) & 1u) == 0u) continue;
            } else {
                const unsigned ent = ulist[q];
                c = (int)(ent / kChunk);
                r = (int)(ent % kChunk);
            }
            return true;
        }
    };
    auto issue = [&](int kind, int c, int r, int slot) {
        volatile ChunkState<NT>& s = tab[c];
        const int e = s.e;
        const unsigned char* w = static_cast<const unsigned char*>(kind == kTaskGate ? a.ex[e].wg : a.ex[e].wu);
        const unsigned char* src = w + (size_t)debug_row(s.jr[r], a.m, a.status) * row_bytes;
        unsigned char* dst = ring + (size_t)(cidx * P + slot) * rc.slot_bytes;
        for (int k = lane; k < row_chunks; k += kWarp) cp_async16(dst + 16 * k, src + 16 * k);
        cp_async_commit();
    };
    auto compute = [&](int kind, int c, int r, int slot) {
        volatile ChunkState<NT>& s = tab[c];
        const int e = s.e;
        const int ntok = sh.es.ntok[e];
        int xt[NT];
#pragma unroll
        for (int k = 0; k < NT; ++k) xt[k] = k < ntok ? (a.route ? sh.es.tok[e][k] : k) : 0;
        float acc[NT];
        smem_row_dot<T, NT>(ring + (size_t)(cidx * P + slot) * rc.slot_bytes, xs, rc.xs_stride, xt, ntok, a.d,
                            lane, acc);
        if (lane == 0) {
            volatile float* dst = kind == kTaskGate ? s.g[r] : s.u[r];
#pragma unroll
            for (int k = 0; k < NT; ++k) dst[k] = acc[k];
        }
        __syncwarp();
    };

    // The weights do not depend on the activations: the first round's rows
    // are set going while the activations are staged, just after the
    // activation loads are issued (so those loads do not queue behind the
    // row copies).
    int qc[kRowsMaxAhead + 1], qr[kRowsMaxAhead + 1];  // claimed rows, oldest first
    int n_q = 0, head_slot = 0;
    const int nr0 = min(kQ4Round, n_local);
    setup(0, nr0);
    named_bar_sync(1, cthreads);
    stage([&]() {
        while (n_q < P && claim(0, kChunk * nr0, qc[n_q], qr[n_q])) {
            issue(kTaskGate, qc[n_q], qr[n_q], n_q);
            ++n_q;
        }
    });

    for (int base = 0; base < n_local; base += kQ4Round) {
        const int nr = min(kQ4Round, n_local - base);
        if (base > 0) {
            setup(base, nr);
            named_bar_sync(1, cthreads);
        }
        for (int phase = 0; phase < 2; ++phase) {
            const int kind = phase == 0 ? kTaskGate : kTaskUp;
            const int n_sub = phase == 0 ? kChunk * nr : sh.q4_ctr[2];
            if (!(base == 0 && phase == 0)) {
                n_q = 0;
                head_slot = 0;
                while (n_q < P && claim(phase, n_sub, qc[n_q], qr[n_q])) {
                    issue(kind, qc[n_q], qr[n_q], n_q);
                    ++n_q;
                }
            }
            while (n_q > 0) {
                cp_async_wait_n<kRowsMaxAhead>(n_q - 1);  // the oldest row has landed
                __syncwarp();
                compute(kind, qc[0], qr[0], head_slot);
                // its slot takes the next row
                for (int i = 1; i < n_q; ++i) {
                    qc[i - 1] = qc[i];
                    qr[i - 1] = qr[i];
                }
                --n_q;
                const int free_slot = head_slot;
                head_slot = head_slot + 1 == P ? 0 : head_slot + 1;
                if (claim(phase, n_sub, qc[n_q], qr[n_q])) {
                    issue(kind, qc[n_q], qr[n_q], free_slot);
                    ++n_q;
                }
            }
            named_bar_sync(1, cthreads);
            if (phase == 0 && cidx == 0) {
                // gate-active rows of each chunk (lane c), listed in chunk order
                unsigned gm = 0u;
                if (lane < nr) {
                    volatile ChunkState<NT>& s = tab[lane];
                    const int ntok = sh.es.ntok[s.e];
                    for (int r = 0; r < kChunk; ++r) {
                        bool ga = false;
                        if (s.jr[r] >= 0) {
#pragma unroll
                            for (int k = 0; k < NT; ++k) ga |= (k < ntok) && (s.g[r][k] > 0.0f);
                        }
                        if (ga) gm |= 1u << r;
                    }
                    s.gmask = gm;
                }
                const int cnt = __popc(gm);
                int incl = cnt;
#pragma unroll
                for (int o = 1; o < kWarp; o <<= 1) {
                    const int v = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += v;
                }
                int pos = incl - cnt;
                for (unsigned m = gm; m; m &= m - 1u) ulist[pos++] = (unsigned short)(lane * kChunk + __ffs(m) - 1);
                if (lane == kWarp - 1) sh.q4_ctr[2] = incl;
                __syncwarp();
            }
            if (phase == 0) named_bar_sync(1, cthreads);
        }
        for (int c0 = cidx * kFinPerWarp; c0 < nr; c0 += C * kFinPerWarp)
            finalize_chunks<NT>(a, sh, tab, c0, min(kFinPerWarp, nr - c0), lane);
        named_bar_sync(1, cthreads);  // the table is refilled next round
    }
}

// PRE: the launch is the predicted stack's (a list made by the kernel just
// before, over a residual that was final before it): the activations are
// staged first and only then is the list waited for. A separate
// instantiation, so that the other launches keep their register budget.
template <typename T, int NT, bool PRE = false>
__global__ void __launch_bounds__(GateUpWarps<NT>::THREADS, 1) k_gate_up_rows(const FfnLaunch a, const RowsCfg rc) {
    constexpr int C = GateUpWarps<NT>::C;
    __shared__ GateUpShared<NT> sh;
    extern __shared__ __align__(128) unsigned char dyn[];
    float* xs = reinterpret_cast<float*>(dyn);  // [NT][xs_stride]
    unsigned char* ring = dyn + (size_t)NT * rc.xs_stride * sizeof(float);  // [C][ahead + 1][slot_bytes]
    ChunkState<NT>* tab =
        reinterpret_cast<ChunkState<NT>*>(ring + (size_t)C * (rc.ahead + 1) * rc.slot_bytes);
    unsigned short* ulist = reinterpret_cast<unsigned short*>(tab + kQ4Round);  // [kQ4Round * kChunk]
    const int n_x = a.route ? a.batch : a.nt;

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) {
        mbar_init(&sh.never, 1);
        for (int q = 0; q < kMaxLocal; ++q) sh.pd.ub[q] = 0;
        mbar_fence_init();
    }
    const bool early = (a.rows == nullptr || a.rows_ready) && a.route == nullptr;
    constexpr bool pre_stage = PRE;
    if (!early && !pre_stage) pdl_wait();
    resolve_experts(a, sh.es);
    pdl_launch_dependents();

    const int n_chunks = (a.n_rows + kChunk - 1) / kChunk;
    const int n_items = sh.es.n_act * n_chunks;
    const int i0 = (int)((long long)n_items * blockIdx.x / gridDim.x);
    const int i1 = (int)((long long)n_items * (blockIdx.x + 1) / gridDim.x);

    if (warp == 0) return;  // the consumer warps copy their own rows
    const int ctid = threadIdx.x - kWarp;
    const int cthreads = C * kWarp;
    const int x_tok0 = a.route ? 0 : a.tok0;
    if (pre_stage) {
        for (int t = 0; t < n_x; ++t) {
            float* xrow = xs + (size_t)t * rc.xs_stride;
            stage_act_row<T>(a.h + (size_t)(x_tok0 + t) * a.d, nullptr, a.d, ctid, cthreads, sh.red,
                             XsPut<T>{xrow});
        }
        named_bar_sync(1, cthreads);
        pdl_wait();
    }
    // Stage the activations; first_rows() (the first weight-row copies) runs
    // once: before the dependency wait when the rows are known without it
    // (no list, or a list written before the launch), else right after the
    // first activation loads are issued.
    auto stage = [&](auto&& first_rows) {
        if (pre_stage) {  // staged already
            first_rows();
            return;
        }
        bool started = false;
        auto once = [&]() {
            if (!started) {
                started = true;
                first_rows();
            }
        };
        if (early) {
            // the weights do not depend on the previous kernel: in a stack this
            // CTA may start while the previous layer's reduction still runs
            // (it lets this kernel be scheduled early), and its first rows
            // stream in meanwhile
            once();
            pdl_wait();
        }
        for (int t = 0; t < n_x; ++t) {
            float* xrow = xs + (size_t)t * rc.xs_stride;
            stage_act_row<T>(a.norm_from_h ? a.h + (size_t)(x_tok0 + t) * a.d : nullptr,
                             static_cast<const T*>(a.x) + (size_t)(x_tok0 + t) * a.d, a.d, ctid, cthreads, sh.red,
                             XsPut<T>{xrow}, once);
        }
        once();
        named_bar_sync(1, cthreads);
    };
    consume_rows<T, NT>(a, sh, ring, xs, tab, ulist, rc, i0, i1, n_chunks, warp - 1, lane, stage);
    // no partial buffer: the caller runs the gathered down kernel after a mask instead
    if (a.partial != nullptr) down_partial<T, NT>(a, sh, i0, i1, n_chunks, warp - 1, lane);
}

// ---------------------------------------------------------------------------
// Fused layer stack: the per-layer chain of Eq. 1-2 for every layer of a
// decode step inside one persistent launch.
//
// One CTA per SM, all co-resident (cooperative launch). Per layer, each CTA
// runs the copy-by-consumer gate+up phases over its chunks and its share of
// the down projection into its partial block, exactly as k_gate_up_rows;
// then, instead of ending the kernel and launching the reduction:
//   grid barrier -> CTA s sums the partial blocks of column slice s (32
//   columns, blocks in CTA order) into the residual -> grid barrier -> the
//   next layer stages rmsnorm(h).
// A grid barrier is one atomic add per CTA on a word whose top bit flips
// once every CTA has arrived; its wait is bounded (kGridWaitLimitNs), after
// which the CTA records kStatusTimeout, raises the abort flag (so the others
// stop at their next barrier instead of waiting out the limit) and returns.
// (Measured alternatives: two-level arrival counters and per-CTA epoch words
// polled by every CTA both made each layer slower.)
// ---------------------------------------------------------------------------
constexpr unsigned long long kGridWaitLimitNs = 4 * kWaitLimitNs;
constexpr int kSliceCols = 32;  // columns a CTA reduces per slice (128 bytes of fp32)

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Grid barrier; consumer threads only (ctid in [0, cthreads)); false when
// the stack must stop. Each CTA adds to one word: CTA 0 adds 2^31 - (grid -
// 1), every other CTA 1, so the word's top bit flips exactly when the last
// CTA arrives, whatever the order, and again at the next barrier. S.bar
// (zero at launch): word 0 the barrier word, word 1 the abort flag.
__device__ bool grid_barrier(const StackLaunch& S, int ctid, int cthreads, int* s_ok) {
    named_bar_sync(1, cthreads);
    if (ctid == 0) {
        int ok = 1;
        __threadfence();
        const unsigned inc = blockIdx.x == 0 ? 0x80000000u - (gridDim.x - 1u) : 1u;
        const unsigned old = atomicAdd(S.bar, inc);
        const unsigned long long t0 = global_ns();
        for (;;) {
            if ((ld_acquire_u32(S.bar) ^ old) & 0x80000000u) break;
            if (ld_acquire_u32(S.bar + 1) != 0u) {
                ok = 0;
                break;
            }
            if (global_ns() - t0 > kGridWaitLimitNs) {
                atomicOr(S.status, kStatusTimeout);
                atomicExch(S.bar + 1, 1u);
                ok = 0;
                break;
            }
        }
        __threadfence();
        *s_ok = ok;
    }
    named_bar_sync(1, cthreads);
    return *s_ok != 0;
}

// h[t][cols of slice s] += sum over the partial blocks of partial[b][t][cols]
// in the order of k_down_reduce, so that the fused stack gives the unfused
// stack's bits: block group g (blocks g, g + 32, g + 64, ...) is summed in
// ascending order, groups 2w and 2w + 1 are added, and those pair sums are
// added for w = 0, 1, ... 15 onto 0. 256 consumer threads = 8 float4 columns
// x 32 block groups.
template <int NT>
__device__ void reduce_slices(const FfnLaunch& a, float* h, int ctid, float4* red) {
    const int d = a.d;
    const int n_slices = (d + kSliceCols - 1) / kSliceCols;
    const int q = ctid & 7;   // float4 column within the slice
    const int gq = ctid >> 3; // block group: blocks gq, gq + 32, ...
    const int nt = a.nt;
    for (int sl = blockIdx.x; sl < n_slices; sl += gridDim.x) {
        const int col = sl * kSliceCols + 4 * q;
        const bool valid = col < d;
        float4 acc[NT];
#pragma unroll
        for (int t = 0; t < NT; ++t) acc[t] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (valid) {
            constexpr int kB = 6;  // blocks in flight per thread
            for (int b0 = gq; b0 < a.partial_ctas; b0 += kB * 32) {
                float4 v[kB][NT];
#pragma unroll
                for (int i = 0; i < kB; ++i) {
                    const int b = b0 + i * 32;
#pragma unroll
                    for (int t = 0; t < NT; ++t)
                        v[i][t] = (b < a.partial_ctas && t < nt)
                                      ? __ldcg(reinterpret_cast<const float4*>(
                                            a.partial + ((size_t)b * a.partial_slots + t) * d + col))
                                      : make_float4(0.f, 0.f, 0.f, 0.f);
                }
#pragma unroll
                for (int i = 0; i < kB; ++i)
#pragma unroll
                    for (int t = 0; t < NT; ++t) {
                        acc[t].x += v[i][t].x;
                        acc[t].y += v[i][t].y;
                        acc[t].z += v[i][t].z;
                        acc[t].w += v[i][t].w;
                    }
            }
        }
#pragma unroll
        for (int t = 0; t < NT; ++t) red[(gq * NT + t) * 8 + q] = acc[t];
        named_bar_sync(1, GateUpWarps<NT>::C * kWarp);
        if (ctid < 8 * NT) {
            const int t = ctid >> 3, qq = ctid & 7;
            const int c = sl * kSliceCols + 4 * qq;
            if (t < nt && c < d) {
                float4 sum = make_float4(0.f, 0.f, 0.f, 0.f);
                for (int w = 0; w < 16; ++w) {
                    const float4 u = red[((2 * w) * NT + t) * 8 + qq];
                    const float4 v = red[((2 * w + 1) * NT + t) * 8 + qq];
                    sum.x += u.x + v.x;
                    sum.y += u.y + v.y;
                    sum.z += u.z + v.z;
                    sum.w += u.w + v.w;
                }
                float4* hp = reinterpret_cast<float4*>(h + (size_t)t * d + c);
                const float4 old = __ldcg(hp);
                *hp = make_float4(old.x + sum.x, old.y + sum.y, old.z + sum.z, old.w + sum.w);
            }
        }
        named_bar_sync(1, GateUpWarps<NT>::C * kWarp);
    }
}

template <int NT>
__global__ void __launch_bounds__(GateUpWarps<NT>::THREADS, 1) k_stack_rows(const StackLaunch S, const RowsCfg rc) {
    using T = __nv_bfloat16;
    constexpr int C = GateUpWarps<NT>::C;
    __shared__ GateUpShared<NT> sh;
    __shared__ FfnLaunch la;  // the current layer's parameters
    __shared__ int s_ok;
    extern __shared__ __align__(128) unsigned char dyn[];
    float* xs = reinterpret_cast<float*>(dyn);
    unsigned char* ring = dyn + (size_t)NT * rc.xs_stride * sizeof(float);
    ChunkState<NT>* tab = reinterpret_cast<ChunkState<NT>*>(ring + (size_t)C * (rc.ahead + 1) * rc.slot_bytes);
    unsigned short* ulist = reinterpret_cast<unsigned short*>(tab + kQ4Round);
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    constexpr int kWords = (int)(sizeof(FfnLaunch) / sizeof(unsigned));
    static_assert(sizeof(FfnLaunch) % sizeof(unsigned) == 0, "FfnLaunch copies as words");

    auto load_layer = [&](int l, int tid, int nthr) {
        const unsigned* src = reinterpret_cast<const unsigned*>(S.layers + l);
        unsigned* dst = reinterpret_cast<unsigned*>(&la);
        for (int i = tid; i < kWords; i += nthr) dst[i] = src[i];
    };
    if (threadIdx.x == 0) {
        mbar_init(&sh.never, 1);
        mbar_fence_init();
    }
    load_layer(0, threadIdx.x, blockDim.x);
    __syncthreads();
    resolve_experts(la, sh.es);  // a single FFN with the same tokens in every layer
    if (warp == 0) return;
    const int ctid = threadIdx.x - kWarp;
    const int cthreads = C * kWarp;

    for (int l = 0; l < S.n_layers; ++l) {
        if (l > 0) {
            load_layer(l, ctid, cthreads);
            named_bar_sync(1, cthreads);
        }
        if (ctid < kMaxLocal) sh.pd.ub[ctid] = 0;
        const int n_chunks = (la.n_rows + kChunk - 1) / kChunk;
        const int i0 = (int)((long long)n_chunks * blockIdx.x / gridDim.x);
        const int i1 = (int)((long long)n_chunks * (blockIdx.x + 1) / gridDim.x);
        auto stage = [&](auto&& first_rows) {
            bool started = false;
            auto once = [&]() {
                if (!started) {
                    started = true;
                    first_rows();
                }
            };
            for (int t = 0; t < la.nt; ++t) {
                float* xrow = xs + (size_t)t * rc.xs_stride;
                stage_act_row<T>(S.h + (size_t)t * la.d, nullptr, la.d, ctid, cthreads, sh.red,
                                 XsPut<T>{xrow}, once);
            }
            once();
            named_bar_sync(1, cthreads);
        };
        consume_rows<T, NT>(la, sh, ring, xs, tab, ulist, rc, i0, i1, n_chunks, warp - 1, lane, stage);
        down_partial<T, NT>(la, sh, i0, i1, n_chunks, warp - 1, lane);
        if (!grid_barrier(S, ctid, cthreads, &s_ok)) return;
        reduce_slices<NT>(la, S.h, ctid, reinterpret_cast<float4*>(ring));
        if (!grid_barrier(S, ctid, cthreads, &s_ok)) return;
    }
}

// Shared memory of the copy-by-consumer kernel: activations, the ring (as
// many rows ahead per warp as fit, up to kRowsMaxAhead), a round's chunk
// states and its list of up rows.
static size_t rows_smem(int elem, int d, int nt, int avail, RowsCfg* rc) {
    rc->xs_stride = (d + 255) / 256 * 256;
    rc->slot_bytes = (d * elem + 127) / 128 * 128;
    const size_t fixed = (size_t)nt * rc->xs_stride * sizeof(float) +
                         (size_t)kQ4Round * sizeof(ChunkState<kAccMaxTokens>) +
                         (size_t)kQ4Round * kChunk * sizeof(unsigned short);
    const int C = GateUpWarps<1>::C;
    int ahead = kRowsMaxAhead;
    while (ahead > 1 && fixed + (size_t)C * (ahead + 1) * rc->slot_bytes > (size_t)avail) --ahead;
    rc->ahead = ahead;
    return fixed + (size_t)C * (ahead + 1) * rc->slot_bytes;
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
int gate_up_config(int wdtype, int d, int x_tokens, int optin_smem, int* slots, int* slot_bytes,
                   int* xs_stride, size_t* smem) {
    const int consumers = x_tokens <= 2 ? GateUpWarps<1>::C : GateUpWarps<8>::C;
    const int row = d * (wdtype == 1 ? 2 : 4);
    *slot_bytes = (row + 127) / 128 * 128;
    *xs_stride = (d + 255) / 256 * 256;
    const size_t xs_bytes = (size_t)x_tokens * (*xs_stride) * sizeof(float);
    const long long avail = (long long)optin_smem - kSmemMargin - (long long)xs_bytes;
    long long s = avail > 0 ? avail / *slot_bytes : 0;
    s = s < kRingBytes / *slot_bytes ? s : kRingBytes / *slot_bytes;
    s = s < kMaxSlots ? s : kMaxSlots;
    // Consumer c takes tasks c, c+C, ...; with S a multiple of C it also owns
    // every use of its slots, so it never waits on a slot whose previous phase
    // belongs to another consumer's unfinished task.
    *slots = (int)(s / consumers * consumers);
    *smem = xs_bytes + (size_t)(*slots) * (*slot_bytes);
    return *slots >= consumers ? 0 : -1;
}

static int g_optin = 0;

template <typename T, int NT>
static cudaError_t launch_t(const FfnLaunch& a, int grid, cudaStream_t stream, bool pdl) {
    const int n_x = a.route ? a.batch : a.nt;
    GateUpCfg cfg;
    size_t smem = 0;
    if (gate_up_config(sizeof(T) == 2 ? 1 : 0, a.d, n_x, g_optin, &cfg.slots, &cfg.slot_bytes,
                       &cfg.xs_stride, &smem) != 0)
        return cudaErrorInvalidValue;
    // a null partial buffer skips the per-CTA down partial (the caller runs
    // the gathered down kernel instead); a given one must hold every CTA
    if (NT <= kAccMaxTokens && a.partial != nullptr && (a.partial_slots < n_x || a.partial_ctas < grid))
        return cudaErrorInvalidValue;
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(grid);
    lc.blockDim = dim3(GateUpWarps<NT>::THREADS);
    lc.dynamicSmemBytes = smem;
    lc.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&lc, k_gate_up<T, NT>, a, cfg);
}

template <int NT>
static cudaError_t launch_mma_t(const FfnLaunch& a, int grid, cudaStream_t stream, bool pdl) {
    MmaCfg mc;
    const size_t smem = mma_smem(a.d, &mc);
    if (smem + kSmemMargin > (size_t)g_optin) return cudaErrorInvalidValue;
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(grid);
    lc.blockDim = dim3(GateUpWarps<NT>::THREADS);
    lc.dynamicSmemBytes = smem;
    lc.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&lc, k_gate_up_mma<NT>, a, mc);
}

template <int NT>
static cudaError_t launch_q4w_t(const FfnLaunch& a, int grid, cudaStream_t stream, bool pdl) {
    MmaCfg mc;
    const size_t smem = q4w_smem(a.d, g_optin - kSmemMargin, &mc);
    if (smem + kSmemMargin > (size_t)g_optin) return cudaErrorInvalidValue;
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(grid);
    lc.blockDim = dim3((kQ4Consumers + 1) * kWarp);
    lc.dynamicSmemBytes = smem;
    lc.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&lc, k_gate_up_q4w<NT>, a, mc);
}

template <typename T, int NT>
static cudaError_t launch_rows_t(const FfnLaunch& a, int grid, cudaStream_t stream, bool pdl) {
    RowsCfg rc;
    const size_t smem = rows_smem((int)sizeof(T), a.d, NT, g_optin - kSmemMargin, &rc);
    if (smem + kSmemMargin > (size_t)g_optin) return cudaErrorInvalidValue;
    const int n_x = a.route ? a.batch : a.nt;
    if (n_x > NT || (a.partial != nullptr && (a.partial_slots < n_x || a.partial_ctas < grid)))
        return cudaErrorInvalidValue;
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(grid);
    lc.blockDim = dim3(GateUpWarps<NT>::THREADS);
    lc.dynamicSmemBytes = smem;
    lc.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = pdl ? 1 : 0;
    if (a.h_ready && a.norm_from_h && a.route == nullptr && a.rows != nullptr && !a.rows_ready)
        return cudaLaunchKernelEx(&lc, k_gate_up_rows<T, NT, true>, a, rc);
    return cudaLaunchKernelEx(&lc, k_gate_up_rows<T, NT, false>, a, rc);
}

template <int NT>
static cudaError_t launch_stack_t(const StackLaunch& S, int d, int grid, cudaStream_t stream) {
    RowsCfg rc;
    const size_t smem = rows_smem(2, d, NT, g_optin - kSmemMargin, &rc);
    if (smem + kSmemMargin > (size_t)g_optin) return cudaErrorInvalidValue;
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(grid);
    lc.blockDim = dim3(GateUpWarps<NT>::THREADS);
    lc.dynamicSmemBytes = smem;
    lc.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;  // every CTA resident at once: the grid barriers rely on it
    attr[0].val.cooperative = 1;
    lc.attrs = attr;
    lc.numAttrs = 1;
    return cudaLaunchKernelEx(&lc, k_stack_rows<NT>, S, rc);
}

int stack_bar_words(int) { return 2; }

bool stack_fused_supported(int d, int nt, int grid, int optin_smem) {
    if (nt < 1 || nt > kAccMaxTokens || grid < 1 || d < 1 || (d * 2) % 16 != 0) return false;
    RowsCfg rc;
    const size_t smem = rows_smem(2, d, nt, optin_smem - kSmemMargin, &rc);
    if (smem + kSmemMargin > (size_t)optin_smem) return false;
    int per_sm = 0, dev = 0, sms = 0;
    const cudaError_t e = nt == 1 ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(
                                        &per_sm, k_stack_rows<1>, GateUpWarps<1>::THREADS, smem)
                                  : cudaOccupancyMaxActiveBlocksPerMultiprocessor(
                                        &per_sm, k_stack_rows<2>, GateUpWarps<2>::THREADS, smem);
    if (e != cudaSuccess || cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return per_sm >= 1 && grid <= per_sm * sms;
}

cudaError_t launch_stack_fused(const StackLaunch& S, int d, int nt, int grid, cudaStream_t stream) {
    if (nt == 1) return launch_stack_t<1>(S, d, grid, stream);
    if (nt == 2) return launch_stack_t<2>(S, d, grid, stream);
    return cudaErrorInvalidValue;
}

// bf16 passes of 1-2 tokens take the copy-by-consumer kernel when its ring fits
static bool use_rows(int wdtype, int d, int pass_tokens) {
    RowsCfg rc;
    return wdtype == 1 && pass_tokens <= kAccMaxTokens &&
           rows_smem(2, d, pass_tokens, g_optin - kSmemMargin, &rc) + kSmemMargin <= (size_t)g_optin;
}

constexpr int kMmaMinTokens = 4;  // narrowest bf16 pass that takes the tensor-core variant

static bool use_mma(int wdtype, int d, int pass_tokens) {
    MmaCfg mc;
    return wdtype == 1 && pass_tokens >= kMmaMinTokens && d % kMmaDAlign == 0 &&
           mma_smem(d, &mc) + kSmemMargin <= (size_t)g_optin;
}

bool int4_supported(int d, int pass_tokens, int optin_smem) {
    MmaCfg mc;
    return d % kMmaDAlign == 0 && pass_tokens >= 1 && pass_tokens <= kAccMaxTokens &&
           q4w_smem(d, optin_smem - kSmemMargin, &mc) + kSmemMargin <= (size_t)optin_smem;
}

template <typename T, int NT>
static cudaError_t prepare_t(int optin) {
    return cudaFuncSetAttribute(k_gate_up<T, NT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                optin - kSmemMargin);
}

cudaError_t prepare_gate_up(int optin_smem) {
    static_assert(sizeof(GateUpShared<2>) + sizeof(FfnLaunch) + 64 < kSmemMargin,
                  "static shared memory of the fused stack exceeds the margin");
    static_assert(sizeof(GateUpShared<8>) < kSmemMargin && sizeof(GateUpShared<4>) < kSmemMargin &&
                      sizeof(GateUpShared<2>) < kSmemMargin && sizeof(GateUpShared<1>) < kSmemMargin,
                  "static shared memory exceeds the margin");
    g_optin = optin_smem;
    cudaError_t e = cudaSuccess;
    if (e == cudaSuccess) e = prepare_t<__nv_bfloat16, 1>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<__nv_bfloat16, 2>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<__nv_bfloat16, 4>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<__nv_bfloat16, 8>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<float, 1>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<float, 2>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<float, 4>(optin_smem);
    if (e == cudaSuccess) e = prepare_t<float, 8>(optin_smem);
    const int dyn = optin_smem - kSmemMargin;
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_gate_up_mma<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_gate_up_mma<8>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_gate_up_rows<__nv_bfloat16, 1, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_gate_up_rows<__nv_bfloat16, 2, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_gate_up_rows<__nv_bfloat16, 1, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_gate_up_rows<__nv_bfloat16, 2, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_stack_rows<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_stack_rows<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_gate_up_q4w<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_gate_up_q4w<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn);
    return e;
}

cudaError_t launch_gate_up(const FfnLaunch& a, int wdtype, int pass_tokens, int grid,
                           cudaStream_t stream, bool pdl) {
    if (wdtype == 2) {
        // INT4 rows: tensor cores, one group per warp, passes of 1-2 tokens
        if (a.d % kMmaDAlign != 0) return cudaErrorInvalidValue;
        if (pass_tokens == 1) return launch_q4w_t<1>(a, grid, stream, pdl);
        if (pass_tokens == 2) return launch_q4w_t<2>(a, grid, stream, pdl);
        return cudaErrorInvalidValue;
    }
    if (use_rows(wdtype, a.d, pass_tokens)) {
        if (pass_tokens == 1) return launch_rows_t<__nv_bfloat16, 1>(a, grid, stream, pdl);
        if (pass_tokens == 2) return launch_rows_t<__nv_bfloat16, 2>(a, grid, stream, pdl);
    }
    if (use_mma(wdtype, a.d, pass_tokens)) {
        if (pass_tokens == 4) return launch_mma_t<4>(a, grid, stream, pdl);
        if (pass_tokens == 8) return launch_mma_t<8>(a, grid, stream, pdl);
    }
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

}  // namespace tsffn
