// ts_wide.cu -- passes of 9-64 tokens (bf16 weights, d a multiple of 256) as
// gathered tensor-core GEMMs that read each weight row once per batch.
//
// At these batch sizes the union of the tokens' active sets covers most
// neurons (Eq. 2 per token, union over the batch), so the FFN of Eq. 1 is a
// dense contraction over the active rows and every row is worth reading once
// for all tokens instead of once per pass of 8:
//   k_wide_gate  G[t][p] = x_t . W_gate[row p]  for every row of the row space,
//                per-token gate bitmaps and their union;
//   k_wide_up    for the union gate-active rows p: u_t,p = x_t . W_up[row p],
//                c_t,p = g_t,p u_t,p where both are positive (Eq. 2), per-token
//                both bitmaps and their union; c is kept as a pair of bf16
//                (hi + lo, |c - hi - lo| <= 2^-16 |c|) for the next product;
//   k_wide_down  partial[s][t][:] = sum over the s-th slice of the union
//                both-active rows p of c_t,p W_down[row p][:] (Eq. 1);
//   k_wide_reduce y_t = sum over slices s in order (or h_t += y_t).
// All products are mma.sync m16n8k16 (bf16 in, fp32 accumulate) on tiles
// staged by 16-byte cp.async through a kStages-deep shared-memory pipeline; row
// tiles are gathered by index, so the sparsity of the union still skips rows.
#include "ts_kernels.cuh"
#include "ts_wide.h"

namespace tsffn {
namespace {

constexpr int kTileK = 64;     // gate/up: K per pipeline stage (128 bytes of a row)
constexpr int kStages = 6;
// gate/up: 8 warps; warp w takes row tiles 3(w%4) .. 3(w%4)+2 over the K-steps
// 2(w/4), 2(w/4)+1 of every stage, and the two halves are added at the end
constexpr int kGuThreads = 256;
constexpr int kTokPad = 64;      // token rows of the activation and c tiles
constexpr int kDownCols = 256;   // down: output columns per CTA
constexpr int kDownK = 32;       // down: rows per pipeline stage
// down: 16 warps; warp w takes columns 32(w%8) .. +31 over K-step w/8 of every stage
constexpr int kDownThreads = 512;
constexpr int kDownPiece = 256;    // down: list rows resolved at a time
constexpr int kScanWords = 2048;   // bitmap words a CTA can scan (m <= 65536)

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
// 16-byte copy global -> shared, zero-filled when `valid` is false
__device__ __forceinline__ void cp16(void* dst, const void* src, bool valid) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_addr(dst)), "l"(src),
                 "r"(valid ? 16 : 0)
                 : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void ldsm4(uint32_t addr, uint32_t (&r)[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}
__device__ __forceinline__ void ldsm2(uint32_t addr, uint32_t& r0, uint32_t& r1) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];" : "=r"(r0), "=r"(r1) : "r"(addr));
}
__device__ __forceinline__ void ldsm4t(uint32_t addr, uint32_t (&r)[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// byte offset of 16-byte chunk c of row r in a tile of 128-byte rows, with
// the chunk index XOR-ed by the row so that 8 rows at one chunk hit 8 banks
__device__ __forceinline__ int swz(int r, int c, int row_bytes) { return r * row_bytes + ((c ^ (r & 7)) << 4); }

// The row of the row space at position p: the list entry or p itself;
// -1 (skipped, recorded) for a list entry out of range or not ascending.
__device__ __forceinline__ int row_of(const WideLaunch& L, int p) {
    if (L.rows == nullptr) return p;
    const int j = L.rows[p];
    if ((unsigned)j >= (unsigned)L.m || (p > 0 && L.rows[p - 1] >= j)) {
        atomicOr(L.status, kStatusBadIndex);
        return -1;
    }
    return j;
}

// Word w of a bitmap of n_bits bits, bits past the end cleared (a bitmap
// shared with longer row spaces of earlier calls may hold stale bits there).
__device__ __forceinline__ unsigned bits_word(const unsigned* words, int w, int n_bits) {
    unsigned v = words[w];
    const int rest = n_bits - w * 32;
    if (rest < 32) v &= (1u << rest) - 1u;
    return v;
}

// Block-wide scan of a bitmap of n_bits bits: every thread learns the number
// of set bits before its own words. Threads own contiguous word ranges.
struct BitScan {
    int w0, w1;     // this thread's words
    int before;     // set bits in words before w0
    int total;      // all set bits
};
template <int THREADS>
__device__ BitScan bit_scan(const unsigned* words, int n_bits, int* s_part) {
    const int tid = threadIdx.x;
    const int n_words = (n_bits + 31) / 32;
    const int per = (n_words + THREADS - 1) / THREADS;
    BitScan b;
    b.w0 = min(tid * per, n_words);
    b.w1 = min(b.w0 + per, n_words);
    int cnt = 0;
    for (int w = b.w0; w < b.w1; ++w) cnt += __popc(bits_word(words, w, n_bits));
    s_part[tid] = cnt;
    __syncthreads();
    // fixed-order prefix over the threads (one warp)
    if (tid < kWarp) {
        int carry = 0;
        for (int base = 0; base < THREADS; base += kWarp) {
            const int v = s_part[base + tid];
            int incl = v;
#pragma unroll
            for (int o = 1; o < kWarp; o <<= 1) {
                const int u = __shfl_up_sync(0xffffffffu, incl, o);
                if (tid >= o) incl += u;
            }
            s_part[base + tid] = carry + incl - v;
            carry += __shfl_sync(0xffffffffu, incl, kWarp - 1);
        }
        if (tid == 0) s_part[THREADS] = carry;
    }
    __syncthreads();
    b.before = s_part[tid];
    b.total = s_part[THREADS];
    __syncthreads();
    return b;
}
// Positions of list entries [i0, i1) (set bits in ascending order) into out[i - i0].
__device__ void bit_emit(const unsigned* words, int n_bits, const BitScan& b, int i0, int i1, int* out) {
    int idx = b.before;
    for (int w = b.w0; w < b.w1 && idx < i1; ++w) {
        unsigned v = bits_word(words, w, n_bits);
        const int n = __popc(v);
        if (idx + n <= i0) {
            idx += n;
            continue;
        }
        while (v) {
            const int bit = __ffs(v) - 1;
            v &= v - 1u;
            if (idx >= i0 && idx < i1) out[idx - i0] = w * 32 + bit;
            ++idx;
        }
    }
}

// ---------------------------------------------------------------------------
// gate / up on the 5th-generation tensor cores: D[i][t] = W[row(i)] . x_t for
// a tile of 128 weight rows (the MMA's M) and all tokens padded to 16 MT (N),
// accumulated in tensor memory.
//
// Every thread copies its share of each K-stage (the 128 gathered weight rows
// and the activations, 128 bytes of each per stage) with 16-byte cp.async
// into a 128-byte-swizzled K-major tile; once a stage has landed everywhere,
// thread 0 issues its four tcgen05.mma (K = 16 each) and a tcgen05.commit
// that arrives on the stage's mbarrier when those MMAs have read the stage.
// The stage is refilled kMmaLag k-blocks later (so the copies never wait on
// the MMA just issued), keeping kStages - kMmaLag stages of copies in
// flight. The accumulator (128 lanes x 16 MT fp32 columns) is read back with
// tcgen05.ld.
// ---------------------------------------------------------------------------
constexpr int kTcRows = 128;  // weight rows per tile: the MMA's M
constexpr int kMmaLag = 2;    // a stage is refilled kMmaLag k-blocks after its MMAs were issued

constexpr int kTcStages = 8;  // most pipeline stages of a tensor-core tile
constexpr int kTcSmem = 192 * 1024;  // pipeline bytes of a tensor-core tile

__device__ __forceinline__ void tc_alloc(uint32_t* dst, uint32_t ncols) {  // warp-wide
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(dst)), "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tc_relinquish() {  // warp-wide
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tc_dealloc(uint32_t taddr, uint32_t ncols) {  // warp-wide
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
// D (tensor memory) = A B^T (+ D when `accumulate`), one thread issues it
__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                       uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// arrive once on `bar` when every tcgen05.mma this thread issued so far has completed
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_addr(bar))
                 : "memory");
}
// 32 lanes x 16 fp32 columns: lane l of the warp gets the 16 columns of TMEM lane (taddr lane + l)
__device__ __forceinline__ void tc_ld16(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
// shared-memory descriptor of a K-major bf16 tile with 128-byte rows and the
// 128-byte swizzle (8-row atoms of 1024 bytes, atom-aligned start)
__device__ __forceinline__ uint64_t sdesc_k128(uint32_t saddr) {
    uint64_t dsc = (uint64_t)((saddr & 0x3FFFFu) >> 4);  // start address, 16-byte units
    dsc |= (uint64_t)1 << 16;                            // leading byte offset (not used by this layout)
    dsc |= (uint64_t)(1024 >> 4) << 32;                  // stride byte offset: between 8-row atoms
    dsc |= (uint64_t)1 << 46;                            // descriptor version
    dsc |= (uint64_t)2 << 61;                            // 128-byte swizzle
    return dsc;
}
// instruction descriptor: bf16 A and B (both K-major), fp32 D, shape M x N
constexpr uint32_t idesc_bf16_f32(int M, int N) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

template <int MT>
struct TcCfg {
    static constexpr int NP = 16 * MT;                 // MMA N: tokens padded to 16
    static constexpr int kA = kTcRows * 128;           // 16 KB of weight rows per stage
    static constexpr int kB = NP * 128;                // activations per stage
    static constexpr int kStage = kA + kB;
    static constexpr int kStages = kTcSmem / kStage > kTcStages ? kTcStages : kTcSmem / kStage;
    static constexpr int kBytes = kStages * kStage + 1024;  // + slack to align the tiles to 1024 bytes
    static constexpr uint32_t kCols = NP <= 16 ? 32 : (NP <= 32 ? 64 : 128);  // tensor-memory columns: a power of 2, >= 2 N
    static constexpr uint32_t kIdesc = idesc_bf16_f32(kTcRows, NP);
    static_assert(NP % 16 == 0 && NP <= 256, "N of an M = 128 MMA");
};

struct TcShared {
    uint64_t mma_done[8];  // per stage: the stage's MMAs have read it
    uint32_t tmem;         // accumulator address
    int fail;
};

// The tile's GEMM into tensor memory; rows_j[i] (shared) is the weight row of
// tile row i (-1: zero). false if a bounded wait ran out (recorded).
template <int MT>
__device__ bool gu_tile_tc(const WideLaunch& L, const __nv_bfloat16* w, const int* rows_j, unsigned char* sm,
                           TcShared& ts) {
    using C = TcCfg<MT>;
    const int tid = threadIdx.x;
    const int d = L.d;
    const int nk = d / kTileK;
    const __nv_bfloat16* wsrc[4];
    int wdst[4];
    bool wok[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int q = tid + kGuThreads * i;  // 1024 chunks: row q / 8, chunk q % 8
        const int r = q >> 3, c = q & 7;
        const int j = rows_j[r];
        wok[i] = j >= 0;
        wsrc[i] = w + (size_t)(j >= 0 ? debug_row(j, L.m, L.status) : 0) * d + c * 8;
        wdst[i] = swz(r, c, 128);
    }
    constexpr int kXPer = (C::NP * 8 + kGuThreads - 1) / kGuThreads;
    const __nv_bfloat16* xsrc[kXPer];
    int xdst[kXPer];
    bool xok[kXPer], xin[kXPer];
#pragma unroll
    for (int i = 0; i < kXPer; ++i) {
        const int q = tid + kGuThreads * i;  // NP x 8 chunks: token q / 8, chunk q % 8
        const int t = q >> 3, c = q & 7;
        xin[i] = t < C::NP;
        xok[i] = t < L.batch;
        xsrc[i] = L.x + (size_t)(t < L.batch ? t : 0) * d + c * 8;
        xdst[i] = C::kA + swz(t, c, 128);
    }
    auto load = [&](int kst, int stage) {
        unsigned char* base = sm + stage * C::kStage;
        const int k0 = kst * kTileK;
#pragma unroll
        for (int i = 0; i < 4; ++i) cp16(base + wdst[i], wsrc[i] + k0, wok[i]);
#pragma unroll
        for (int i = 0; i < kXPer; ++i)
            if (xin[i]) cp16(base + xdst[i], xsrc[i] + k0, xok[i]);
    };
    const uint32_t sm0 = smem_addr(sm);
    constexpr int S = C::kStages, D = kMmaLag;
    bool ok = true;
#pragma unroll 1
    for (int s = 0; s < S - D; ++s) {
        if (s < nk) load(s, s);
        cp_commit();
    }
    for (int kst = 0; kst < nk; ++kst) {
        cp_wait<S - D - 1>();      // k-block kst has landed (this thread's copies)
        fence_proxy_async_smem();  // ... and is visible to the tensor cores
        __syncthreads();
        if (ts.fail) {             // a bounded wait ran out somewhere (set before the barrier)
            ok = false;
            break;
        }
        if (tid == 0) {
            tc_fence_after();
            const uint32_t a0 = sm0 + (kst % S) * C::kStage;
            const uint64_t ad = sdesc_k128(a0), bd = sdesc_k128(a0 + C::kA);
#pragma unroll
            for (int kk = 0; kk < kTileK / 16; ++kk)  // 32 bytes of each row per MMA
                tc_mma(ts.tmem, ad + 2 * kk, bd + 2 * kk, C::kIdesc, (kst | kk) != 0);
            tc_commit(&ts.mma_done[kst % S]);
        }
        // refill the stage of k-block kst - D, whose MMAs were issued D
        // iterations ago, so the wait rarely stalls on the MMA pipeline
        const int nxt = kst + S - D;
        if (nxt < nk) {
            if (kst >= D && !mbar_wait(&ts.mma_done[(kst - D) % S], (unsigned)((kst - D) / S) & 1u)) ts.fail = 1;
            load(nxt, nxt % S);
        }
        cp_commit();
    }
    // every MMA done (the last commit covers all earlier ones)
    if (ok && !mbar_wait(&ts.mma_done[(nk - 1) % S], (unsigned)((nk - 1) / S) & 1u)) ts.fail = 1;
    cp_wait<0>();
    __syncthreads();
    ok = ok && ts.fail == 0;
    if (!ok && tid == 0) atomicOr(L.status, kStatusTimeout);
    tc_fence_after();
    return ok;
}

// tensor memory and barriers for the tile; warp 0 allocates
template <int MT>
__device__ void tc_setup(TcShared& ts) {
    if (threadIdx.x < kWarp) {
        tc_alloc(&ts.tmem, TcCfg<MT>::kCols);
        tc_relinquish();
    }
    if (threadIdx.x == 0) {
        for (int s = 0; s < TcCfg<MT>::kStages; ++s) mbar_init(&ts.mma_done[s], 1);
        ts.fail = 0;
        mbar_fence_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
}
template <int MT>
__device__ void tc_teardown(TcShared& ts) {
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x < kWarp) {
        tc_fence_after();
        tc_dealloc(ts.tmem, TcCfg<MT>::kCols);
    }
}

__device__ __forceinline__ unsigned char* align1024(unsigned char* p) {
    const uint32_t a = smem_addr(p);
    return p + ((1024u - (a & 1023u)) & 1023u);
}

template <int MT>
__global__ void __launch_bounds__(kGuThreads) k_wide_gate(const WideLaunch L) {
    extern __shared__ __align__(1024) unsigned char sm_raw[];
    __shared__ int rows_j[kTcRows];
    __shared__ unsigned s_union[kTcRows / 32];
    __shared__ TcShared ts;
    unsigned char* sm = align1024(sm_raw);
    pdl_wait();
    pdl_launch_dependents();
    const int p0 = blockIdx.x * kTcRows;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid < kTcRows) rows_j[tid] = p0 + tid < L.n_rows ? row_of(L, p0 + tid) : -1;
    if (tid < kTcRows / 32) s_union[tid] = 0u;
    tc_setup<MT>(ts);
    const bool ok = gu_tile_tc<MT>(L, L.wg, rows_j, sm, ts);
    // warp w reads tile rows 32 (w % 4) .. + 31, token tiles w / 4, w / 4 + 2
    const int q = warp & 3, i = 32 * q + lane, p = p0 + i;
    const int n_in = min(kTcRows, L.n_rows - p0);
    const bool row_in = i < n_in && rows_j[i] >= 0;
    unsigned uw = 0u;
    const int word = (p0 + 32 * q) / 32;  // bitmap word of rows p0 + 32 q .. + 31
    const bool word_in = p0 + 32 * q < L.n_rows;
    if (ok) {
        for (int mt = warp >> 2; mt < MT; mt += 2) {
            float v[16];
            tc_ld16(ts.tmem + ((uint32_t)(32 * q) << 16) + 16 * mt, v);
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const int t = 16 * mt + e;
                if (t < L.batch && i < n_in) L.gval[(size_t)t * L.n_rows + p] = v[e];
                const unsigned bits = __ballot_sync(0xffffffffu, t < L.batch && row_in && v[e] > 0.0f);
                if (t < L.batch && lane == 0 && word_in) {
                    reinterpret_cast<unsigned*>(L.gbits + (size_t)t * L.nbytes)[word] = bits;
                    reinterpret_cast<unsigned*>(L.bbits + (size_t)t * L.nbytes)[word] = 0u;
                }
                uw |= bits;
            }
        }
        if (lane == 0 && uw) atomicOr(&s_union[q], uw);
    }
    __syncthreads();
    if (ok && warp < 4 && lane == 0 && word_in) {
        reinterpret_cast<unsigned*>(L.ugbits)[word] = s_union[q];
        reinterpret_cast<unsigned*>(L.ubits)[word] = 0u;
    }
    tc_teardown<MT>(ts);
}

template <int MT>
__global__ void __launch_bounds__(kGuThreads) k_wide_up(const WideLaunch L) {
    extern __shared__ __align__(1024) unsigned char sm_raw[];
    __shared__ int rows_j[kTcRows];
    __shared__ int pos[kTcRows];
    __shared__ int s_part[kGuThreads + 1];
    __shared__ TcShared ts;
    unsigned char* sm = align1024(sm_raw);
    pdl_wait();
    pdl_launch_dependents();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const unsigned* ug = reinterpret_cast<const unsigned*>(L.ugbits);
    const BitScan bs = bit_scan<kGuThreads>(ug, L.n_rows, s_part);
    const int i0 = blockIdx.x * kTcRows;
    if (i0 >= bs.total) return;  // the union gate-active list is shorter
    const int n_in = min(kTcRows, bs.total - i0);
    if (tid < kTcRows) pos[tid] = -1;
    __syncthreads();
    bit_emit(ug, L.n_rows, bs, i0, i0 + n_in, pos);
    __syncthreads();
    if (tid < kTcRows) rows_j[tid] = pos[tid] >= 0 ? (L.rows ? L.rows[pos[tid]] : pos[tid]) : -1;
    tc_setup<MT>(ts);
    const bool ok = gu_tile_tc<MT>(L, L.wu, rows_j, sm, ts);
    // c = g u where both are positive (Eq. 2), split into bf16 hi + lo
    const int q = warp & 3, i = 32 * q + lane;
    const int p = pos[i];
    unsigned* bb = reinterpret_cast<unsigned*>(L.bbits);
    unsigned* ub = reinterpret_cast<unsigned*>(L.ubits);
    if (ok) {
      // A warp whose 32 rows fill one bitmap word (the list is dense there:
      // nearly every neuron gate-active) ORs its bits together, so the word
      // takes one atomic per token instead of 32 contending ones; elsewhere
      // one atomic per both-active (row, token) measured faster.
      const int w32 = p >= 0 ? p / 32 : -1;
      const unsigned same = __match_any_sync(0xffffffffu, w32);
      if (same == 0xffffffffu && w32 >= 0) {
        const unsigned bit = 1u << (p % 32);
        const bool leader = (__ffs(same) - 1) == lane;
        unsigned any_both = 0u;
        for (int mt = warp >> 2; mt < kTokPad / 16; mt += 2) {
            float v[16];
            if (mt < MT) tc_ld16(ts.tmem + ((uint32_t)(32 * q) << 16) + 16 * mt, v);
            __align__(16) __nv_bfloat16 hi[16], lo[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const int t = 16 * mt + e;
                float c = 0.0f;
                if (p >= 0 && mt < MT && t < L.batch) {
                    const float gv = L.gval[(size_t)t * L.n_rows + p];
                    const float uv = v[e];
                    if (gv > 0.0f && uv > 0.0f) c = gv * uv;
                }
                const unsigned mine = c > 0.0f ? bit : 0u;
                any_both |= mine;
                if (mt < MT && t < L.batch) {
                    const unsigned word_bits = __reduce_or_sync(same, mine);
                    if (leader && word_bits) atomicOr(bb + (size_t)t * (L.nbytes / 4) + w32, word_bits);
                }
                hi[e] = __float2bfloat16_rn(c);
                lo[e] = __float2bfloat16_rn(c - __bfloat162float(hi[e]));
            }
            if (p < 0) continue;
            uint4* dh = reinterpret_cast<uint4*>(L.c_hi + (size_t)p * kTokPad + 16 * mt);
            uint4* dl = reinterpret_cast<uint4*>(L.c_lo + (size_t)p * kTokPad + 16 * mt);
            dh[0] = reinterpret_cast<const uint4*>(hi)[0];
            dh[1] = reinterpret_cast<const uint4*>(hi)[1];
            dl[0] = reinterpret_cast<const uint4*>(lo)[0];
            dl[1] = reinterpret_cast<const uint4*>(lo)[1];
        }
        const unsigned union_bits = __reduce_or_sync(same, any_both);
        if (leader && union_bits) atomicOr(ub + w32, union_bits);
      } else {
        for (int mt = warp >> 2; mt < kTokPad / 16; mt += 2) {
            float v[16];
            if (mt < MT) tc_ld16(ts.tmem + ((uint32_t)(32 * q) << 16) + 16 * mt, v);
            if (p < 0) continue;
            __align__(16) __nv_bfloat16 hi[16], lo[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const int t = 16 * mt + e;
                float c = 0.0f;
                if (mt < MT && t < L.batch) {
                    const float gv = L.gval[(size_t)t * L.n_rows + p];
                    const float uv = v[e];
                    if (gv > 0.0f && uv > 0.0f) {
                        c = gv * uv;
                        atomicOr(bb + (size_t)t * (L.nbytes / 4) + p / 32, 1u << (p % 32));
                        atomicOr(ub + p / 32, 1u << (p % 32));
                    }
                }
                hi[e] = __float2bfloat16_rn(c);
                lo[e] = __float2bfloat16_rn(c - __bfloat162float(hi[e]));
            }
            uint4* dh = reinterpret_cast<uint4*>(L.c_hi + (size_t)p * kTokPad + 16 * mt);
            uint4* dl = reinterpret_cast<uint4*>(L.c_lo + (size_t)p * kTokPad + 16 * mt);
            dh[0] = reinterpret_cast<const uint4*>(hi)[0];
            dh[1] = reinterpret_cast<const uint4*>(hi)[1];
            dl[0] = reinterpret_cast<const uint4*>(lo)[0];
            dl[1] = reinterpret_cast<const uint4*>(lo)[1];
        }
      }
    }
    tc_teardown<MT>(ts);
}

// ---------------------------------------------------------------------------
// down: partial[s][t][n0 .. n0+255] over slice s of the union both-active rows
// ---------------------------------------------------------------------------
struct DnSmem {
    static constexpr int kW = kDownK * kDownCols * 2;  // 16 KB per stage
    static constexpr int kC = kDownK * kTokPad * 2;    // 4 KB per stage (hi or lo)
    static constexpr int kStage = kW + 2 * kC;
    static constexpr int kBytes = kStages * kStage;    // 96 KB
};

template <int MT>
__global__ void __launch_bounds__(kDownThreads) k_wide_down(const WideLaunch L) {
    extern __shared__ __align__(128) unsigned char sm[];
    __shared__ int pos[kDownPiece];
    __shared__ int s_part[kDownThreads + 1];
    pdl_wait();
    pdl_launch_dependents();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int d = L.d;
    const int n_tiles = d / kDownCols;
    const int n0 = (blockIdx.x % n_tiles) * kDownCols;
    const int s = blockIdx.x / n_tiles;
    const unsigned* ub = reinterpret_cast<const unsigned*>(L.ubits);
    const BitScan bs = bit_scan<kDownThreads>(ub, L.n_rows, s_part);
    const int k_begin = (int)((long long)bs.total * s / L.ks);
    const int k_end = (int)((long long)bs.total * (s + 1) / L.ks);

    float acc[MT][4][4];
#pragma unroll
    for (int a = 0; a < MT; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b)
#pragma unroll
            for (int e = 0; e < 4; ++e) acc[a][b][e] = 0.0f;

    for (int piece = k_begin; piece < k_end; piece += kDownPiece) {
        const int n_piece = min(kDownPiece, k_end - piece);
        __syncthreads();  // the previous piece's positions are no longer read
        for (int i = tid; i < kDownPiece; i += kDownThreads) pos[i] = -1;
        __syncthreads();
        bit_emit(ub, L.n_rows, bs, piece, piece + n_piece, pos);
        __syncthreads();
        const int nk = (n_piece + kDownK - 1) / kDownK;
        // this thread's copies per stage: 2 weight chunks (32 rows x 32), 1 hi or lo chunk (32 rows x 8)
        auto load = [&](int kst, int stage) {
            unsigned char* base = sm + stage * DnSmem::kStage;
#pragma unroll
            for (int i = 0; i < 2; ++i) {
                const int q = tid + kDownThreads * i;  // 1024 chunks: row q / 32, chunk q % 32
                const int r = q >> 5, c = q & 31;
                const int li = kst * kDownK + r;
                const int p = li < n_piece ? pos[li] : -1;
                const int j = debug_row(p >= 0 ? (L.rows ? L.rows[p] : p) : 0, L.m, L.status);
                cp16(base + r * (kDownCols * 2) + (((c & ~7) | ((c ^ r) & 7)) << 4),
                     L.wd + (size_t)j * d + n0 + c * 8, p >= 0);
            }
            {
                const int q = tid & 255, lo = tid >> 8;  // 2 x 256 chunks: row q / 8, chunk q % 8
                const int r = q >> 3, c = q & 7;
                const int li = kst * kDownK + r;
                const int p = li < n_piece ? pos[li] : -1;
                const size_t off = (size_t)(p >= 0 ? p : 0) * kTokPad + c * 8;
                cp16(base + DnSmem::kW + lo * DnSmem::kC + swz(r, c, 128), (lo ? L.c_lo : L.c_hi) + off, p >= 0);
            }
        };
#pragma unroll
        for (int st = 0; st < kStages - 1; ++st) {
            if (st < nk) load(st, st);
            cp_commit();
        }
        for (int kst = 0; kst < nk; ++kst) {
            cp_wait<kStages - 2>();
            __syncthreads();
            if (kst + kStages - 1 < nk) load(kst + kStages - 1, (kst + kStages - 1) % kStages);
            cp_commit();
            const uint32_t wsa = smem_addr(sm + (kst % kStages) * DnSmem::kStage);
            const uint32_t cha = wsa + DnSmem::kW;
            const uint32_t cla = cha + DnSmem::kC;
            {
                const int kk = warp >> 3;  // this warp's K-step of the stage
                // A (tokens x k) from the stored [k][token] c tile, transposed:
                // a0 (tok 0-7, k 0-7), a1 (tok 8-15, k 0-7), a2 (tok 0-7, k 8-15), a3 (tok 8-15, k 8-15)
                uint32_t ah[MT][4], al[MT][4];
                const int kr = kk * 16 + ((lane >> 4) << 3) + (lane & 7);
#pragma unroll
                for (int mt = 0; mt < MT; ++mt) {
                    const int c = mt * 2 + ((lane >> 3) & 1);
                    ldsm4t(cha + swz(kr, c, 128), ah[mt]);
                    ldsm4t(cla + swz(kr, c, 128), al[mt]);
                }
                // B (k x columns) from the stored [k][column] W_down tile, transposed:
                // per column tile of 8: b0 (k 0-7), b1 (k 8-15)
                uint32_t bw[2][4];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int c = (warp & 7) * 4 + h * 2 + (lane >> 4);  // 16-byte chunk = 8 columns
                    const int r = kk * 16 + (((lane >> 3) & 1) << 3) + (lane & 7);
                    ldsm4t(wsa + r * (kDownCols * 2) + (((c & ~7) | ((c ^ r) & 7)) << 4), bw[h]);
                }
#pragma unroll
                for (int mt = 0; mt < MT; ++mt)
#pragma unroll
                    for (int nt = 0; nt < 4; ++nt) {
                        const uint32_t b0 = bw[nt >> 1][(nt & 1) * 2], b1 = bw[nt >> 1][(nt & 1) * 2 + 1];
                        mma16816(acc[mt][nt], ah[mt], b0, b1);
                        mma16816(acc[mt][nt], al[mt], b0, b1);
                    }
            }
        }
        cp_wait<0>();
    }
    // the two K-step halves of each column group added in a fixed order,
    // then the slice's partial sums for tokens < batch
    __syncthreads();
    float* red = reinterpret_cast<float*>(sm);  // [8 groups][MT][4][4][32 lanes]
    const int grp = warp & 7;
    if (warp >= 8) {
#pragma unroll
        for (int mt = 0; mt < MT; ++mt)
#pragma unroll
            for (int nt = 0; nt < 4; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) red[(((grp * MT + mt) * 4 + nt) * 4 + e) * kWarp + lane] = acc[mt][nt][e];
    }
    __syncthreads();
    if (warp >= 8) return;
    const int g = lane >> 2, t4 = lane & 3;
    float* ps = L.partial + (size_t)s * L.batch * d;
#pragma unroll
    for (int mt = 0; mt < MT; ++mt)
#pragma unroll
        for (int nt = 0; nt < 4; ++nt) {
            float v[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) v[e] = acc[mt][nt][e] + red[(((grp * MT + mt) * 4 + nt) * 4 + e) * kWarp + lane];
            const int col = n0 + grp * 32 + nt * 8 + 2 * t4;
            const int tok = mt * 16 + g;
            if (tok < L.batch) *reinterpret_cast<float2*>(ps + (size_t)tok * d + col) = make_float2(v[0], v[1]);
            if (tok + 8 < L.batch)
                *reinterpret_cast<float2*>(ps + (size_t)(tok + 8) * d + col) = make_float2(v[2], v[3]);
        }
}

// ---------------------------------------------------------------------------
// down on the 5th-generation tensor cores: D[n][t] = sum over the slice's
// union both-active rows p of W_down[row p][n0 + n] c_t,p, for 128 output
// columns (the MMA's M) and all tokens (N), both operands MN-major: a K-row
// of the A tile is 256 contiguous bytes of a W_down row, a K-row of the B
// tile the 128 bytes of c (64 tokens) of that row. c enters twice, as its
// bf16 hi and lo parts, into the same accumulator.
// Stage (64 list rows): A as two 64-column halves of 64 rows x 128 bytes
// (128-byte swizzle, 8-row atoms), then the c hi and lo tiles (64 rows x
// 128 bytes each).
// ---------------------------------------------------------------------------
constexpr int kTcDownCols = 128;  // output columns per CTA: the MMA's M
constexpr int kTcDownK = 64;      // list rows per stage
constexpr int kTcDownPiece = 2048;  // list entries resolved at a time

template <int MT>
struct TcDownCfg {
    static constexpr int NP = 16 * MT;
    static constexpr int kAHalf = kTcDownK * 128;  // 8 KB: 64 rows x 64 columns
    static constexpr int kA = 2 * kAHalf;
    static constexpr int kC = kTcDownK * 128;      // 8 KB: 64 rows x 64 tokens
    static constexpr int kStage = kA + 2 * kC;     // 32 KB
    static constexpr int kStages = kTcSmem / kStage > kTcStages ? kTcStages : kTcSmem / kStage;
    static constexpr int kBytes = kStages * kStage + 1024;
    static constexpr uint32_t kCols = NP <= 16 ? 32 : (NP <= 32 ? 64 : 128);
    // bf16 A and B, both MN-major (bits 15, 16), fp32 D, M = 128, N = NP
    static constexpr uint32_t kIdesc = idesc_bf16_f32(kTcDownCols, NP) | (1u << 15) | (1u << 16);
};

// MN-major tile with the 128-byte swizzle: 64 contiguous MN elements per
// 128-byte K-row, 8 K-rows per 1024-byte atom; `lbo` bytes between 64-element
// MN blocks, 1024 bytes between 8-row K groups
__device__ __forceinline__ uint64_t sdesc_mn128(uint32_t saddr, uint32_t lbo) {
    uint64_t dsc = (uint64_t)((saddr & 0x3FFFFu) >> 4);
    dsc |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    dsc |= (uint64_t)(1024 >> 4) << 32;
    dsc |= (uint64_t)1 << 46;
    dsc |= (uint64_t)2 << 61;
    return dsc;
}

template <int MT>
__global__ void __launch_bounds__(kGuThreads) k_wide_down_tc(const WideLaunch L) {
    using C = TcDownCfg<MT>;
    extern __shared__ __align__(1024) unsigned char sm_raw[];
    __shared__ int pos[kTcDownPiece];
    __shared__ int s_part[kGuThreads + 1];
    __shared__ TcShared ts;
    unsigned char* sm = align1024(sm_raw);
    pdl_wait();
    pdl_launch_dependents();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int d = L.d;
    const int n_tiles = d / kTcDownCols;
    const int n0 = (blockIdx.x % n_tiles) * kTcDownCols;
    const int sl = blockIdx.x / n_tiles;
    const unsigned* ub = reinterpret_cast<const unsigned*>(L.ubits);
    const BitScan bs = bit_scan<kGuThreads>(ub, L.n_rows, s_part);
    const int k_begin = (int)((long long)bs.total * sl / L.ks);
    const int k_end = (int)((long long)bs.total * (sl + 1) / L.ks);
    const int n_list = k_end - k_begin;
    const int nk = (n_list + kTcDownK - 1) / kTcDownK;
    float* ps = L.partial + (size_t)sl * L.batch * d;
    const int q = warp & 3, col = n0 + 32 * q + lane;
    if (nk == 0) {
        // an empty slice still writes its partial (zeros)
        for (int t = warp >> 2; t < L.batch; t += 2) ps[(size_t)t * d + col] = 0.0f;
        return;
    }
    tc_setup<MT>(ts);
    int piece = -1;  // list entries [piece * kTcDownPiece, +kTcDownPiece) of the slice are in pos[]
    auto resolve = [&](int pc) {
        __syncthreads();  // nobody reads the previous piece any more
        const int e0 = k_begin + pc * kTcDownPiece;
        const int e1 = min(k_end, e0 + kTcDownPiece);
        for (int i = tid; i < kTcDownPiece; i += kGuThreads) pos[i] = -1;
        __syncthreads();
        bit_emit(ub, L.n_rows, bs, e0, e1, pos);
        __syncthreads();
        piece = pc;
    };
    auto load = [&](int kb, int stage) {
        unsigned char* base = sm + stage * C::kStage;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            // W_down: 64 rows x 16 chunks of 8 columns
            const int qq = tid + kGuThreads * i;
            const int r = qq >> 4, c16 = qq & 15;
            const int li = kb * kTcDownK + r;
            const int pp = li < n_list ? pos[li - piece * kTcDownPiece] : -1;
            const int j = debug_row(pp >= 0 ? (L.rows ? L.rows[pp] : pp) : 0, L.m, L.status);
            const int h = c16 >> 3, c = c16 & 7;
            cp16(base + h * C::kAHalf + swz(r, c, 128), L.wd + (size_t)j * d + n0 + c16 * 8, pp >= 0);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            // c hi / lo: 64 rows x 8 chunks of 8 tokens each
            const int qq = tid + kGuThreads * i;
            const int lo = qq >> 9, r = (qq >> 3) & 63, c = qq & 7;
            const int li = kb * kTcDownK + r;
            const int pp = li < n_list ? pos[li - piece * kTcDownPiece] : -1;
            const size_t off = (size_t)(pp >= 0 ? pp : 0) * kTokPad + c * 8;
            cp16(base + C::kA + lo * C::kC + swz(r, c, 128), (lo ? L.c_lo : L.c_hi) + off, pp >= 0);
        }
    };
    auto ensure_piece = [&](int kb) {
        const int pc = kb * kTcDownK / kTcDownPiece;
        if (pc != piece) resolve(pc);
    };
    const uint32_t sm0 = smem_addr(sm);
    constexpr int S = C::kStages, D = kMmaLag;
    bool ok = true;
    for (int s = 0; s < S - D; ++s) {
        if (s < nk) {
            ensure_piece(s);
            load(s, s);
        }
        cp_commit();
    }
    for (int kb = 0; kb < nk; ++kb) {
        cp_wait<S - D - 1>();
        fence_proxy_async_smem();
        __syncthreads();
        if (ts.fail) {
            ok = false;
            break;
        }
        if (tid == 0) {
            tc_fence_after();
            const uint32_t a0 = sm0 + (kb % S) * C::kStage;
            const uint32_t b0 = a0 + C::kA;
#pragma unroll
            for (int kk = 0; kk < kTcDownK / 16; ++kk) {  // 16 rows = two 8-row atoms per MMA
                const uint64_t ad = sdesc_mn128(a0 + kk * 2048, C::kAHalf);
                tc_mma(ts.tmem, ad, sdesc_mn128(b0 + kk * 2048, C::kC), C::kIdesc, (kb | kk) != 0);
                tc_mma(ts.tmem, ad, sdesc_mn128(b0 + C::kC + kk * 2048, C::kC), C::kIdesc, 1u);
            }
            tc_commit(&ts.mma_done[kb % S]);
        }
        const int nxt = kb + S - D;
        if (nxt < nk) {
            if (kb >= D && !mbar_wait(&ts.mma_done[(kb - D) % S], (unsigned)((kb - D) / S) & 1u)) ts.fail = 1;
            ensure_piece(nxt);
            load(nxt, nxt % S);
        }
        cp_commit();
    }
    if (ok && !mbar_wait(&ts.mma_done[(nk - 1) % S], (unsigned)((nk - 1) / S) & 1u)) ts.fail = 1;
    cp_wait<0>();
    __syncthreads();
    ok = ok && ts.fail == 0;
    if (!ok && tid == 0) atomicOr(L.status, kStatusTimeout);
    tc_fence_after();
    if (ok) {
        // warp w: columns n0 + 32 (w % 4) + lane, token tiles w / 4, w / 4 + 2
        for (int mt = warp >> 2; mt < MT; mt += 2) {
            float v[16];
            tc_ld16(ts.tmem + ((uint32_t)(32 * q) << 16) + 16 * mt, v);
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const int t = 16 * mt + e;
                if (t < L.batch) ps[(size_t)t * d + col] = v[e];
            }
        }
    }
    tc_teardown<MT>(ts);
}

// y_t = sum of the slices' partials in slice order (or h_t += y_t)
__global__ void __launch_bounds__(256) k_wide_reduce(const WideLaunch L) {
    pdl_wait();
    pdl_launch_dependents();
    const size_t n = (size_t)L.batch * L.d;
    const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    float v = 0.0f;
    for (int s = 0; s < L.ks; ++s) v += L.partial[(size_t)s * n + i];
    if (L.residual_out)
        L.h[i] += v;
    else
        L.y[i] = v;
}

// x_t = bf16(h_t / sqrt(mean(h_t^2) + 1e-5)) with x[d-1] = 1 (the stack glue),
// one CTA per token, the same reduction order as the gate+up kernels' staging
__global__ void __launch_bounds__(256) k_wide_norm(const WideLaunch L, const float* h, __nv_bfloat16* xout) {
    __shared__ float red[8];
    pdl_wait();
    pdl_launch_dependents();
    const int t = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const float* hr = h + (size_t)t * L.d;
    float ss = 0.0f;
    for (int i = tid; i < L.d; i += 256) ss = fmaf(hr[i], hr[i], ss);
    ss = warp_sum(ss);
    if (lane == 0) red[warp] = ss;
    __syncthreads();
    float tot = 0.0f;
    for (int w = 0; w < 8; ++w) tot += red[w];
    const float rms = __fsqrt_rn(__fadd_rn(__fdiv_rn(tot, (float)L.d), 1e-5f));
    for (int i = tid; i < L.d; i += 256)
        xout[(size_t)t * L.d + i] = __float2bfloat16_rn(i == L.d - 1 ? 1.0f : __fdiv_rn(hr[i], rms));
}

template <typename K>
cudaError_t launch(K kernel, int grid, int threads, size_t smem, cudaStream_t stream, bool pdl, const WideLaunch& L) {
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(grid);
    lc.blockDim = dim3(threads);
    lc.dynamicSmemBytes = smem;
    lc.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&lc, kernel, L);
}

// The tensor-core down kernel (128-column tiles) for passes of more than 48
// tokens; the mma.sync one (256-column tiles, half the c traffic per weight
// byte) below that, where it measured faster.
constexpr bool tc_down(int mt) { return mt >= 4; }

template <int MT>
cudaError_t run_t(const WideLaunch& L0, cudaStream_t stream, bool pdl) {
    WideLaunch L = L0;
    // the tensor-core down kernel's column tiles are half as wide: half as
    // many slices keep its grid at about one CTA per SM (the reduction sums
    // the same count)
    if (tc_down(MT)) L.ks = L0.ks * kTcDownCols / kDownCols > 0 ? L0.ks * kTcDownCols / kDownCols : 1;
    const int gu_grid = (L.n_rows + kTcRows - 1) / kTcRows;
    cudaError_t e = launch(k_wide_gate<MT>, gu_grid, kGuThreads, TcCfg<MT>::kBytes, stream, pdl, L);
    if (e == cudaSuccess) e = launch(k_wide_up<MT>, gu_grid, kGuThreads, TcCfg<MT>::kBytes, stream, true, L);
    if (e == cudaSuccess) {
        if (tc_down(MT))
            e = launch(k_wide_down_tc<MT>, (L.d / kTcDownCols) * L.ks, kGuThreads, TcDownCfg<MT>::kBytes, stream,
                       true, L);
        else
            e = launch(k_wide_down<MT>, (L.d / kDownCols) * L.ks, kDownThreads, DnSmem::kBytes, stream, true, L);
    }
    if (e == cudaSuccess) {
        const int n = L.batch * L.d;
        e = launch(k_wide_reduce, (n + 255) / 256, 256, 0, stream, true, L);
    }
    return e;
}

template <int MT>
cudaError_t prepare_t() {
    cudaError_t e = cudaFuncSetAttribute(k_wide_gate<MT>, cudaFuncAttributeMaxDynamicSharedMemorySize, TcCfg<MT>::kBytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_wide_up<MT>, cudaFuncAttributeMaxDynamicSharedMemorySize, TcCfg<MT>::kBytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_wide_down<MT>, cudaFuncAttributeMaxDynamicSharedMemorySize, DnSmem::kBytes);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_wide_down_tc<MT>, cudaFuncAttributeMaxDynamicSharedMemorySize, TcDownCfg<MT>::kBytes);
    return e;
}

}  // namespace

bool wide_supported(int wdtype, int d, int m, int batch) {
    return wdtype == 1 && batch > kMaxPass && batch <= kTokPad && d % kDownCols == 0 && m <= kScanWords * 32;
}

int wide_slices(int d, int num_sms) {
    // enough slices for either down kernel (the tensor-core one has narrower column tiles)
    const int n_tiles = d / kDownCols;
    return n_tiles >= num_sms ? 1 : num_sms / n_tiles;
}

cudaError_t prepare_wide() {
    cudaError_t e = prepare_t<1>();
    if (e == cudaSuccess) e = prepare_t<2>();
    if (e == cudaSuccess) e = prepare_t<3>();
    if (e == cudaSuccess) e = prepare_t<4>();
    return e;
}

cudaError_t launch_wide(const WideLaunch& L, cudaStream_t stream, bool pdl) {
    switch ((L.batch + 15) / 16) {
        case 1: return run_t<1>(L, stream, pdl);
        case 2: return run_t<2>(L, stream, pdl);
        case 3: return run_t<3>(L, stream, pdl);
        case 4: return run_t<4>(L, stream, pdl);
    }
    return cudaErrorInvalidValue;
}

cudaError_t launch_wide_norm(const WideLaunch& L, const float* h, __nv_bfloat16* xout, cudaStream_t stream, bool pdl) {
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(L.batch);
    lc.blockDim = dim3(256);
    lc.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&lc, k_wide_norm, L, h, xout);
}

}  // namespace tsffn
