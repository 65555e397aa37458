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

constexpr int kTileRows = 96;  // gate/up: weight rows per CTA
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
// gate / up: C[t][i] = x_t . W[row(i)] for a tile of 96 rows, all tokens
// ---------------------------------------------------------------------------
struct GuSmem {
    static constexpr int kX = kTokPad * kTileK * 2;     // 8 KB per stage
    static constexpr int kW = kTileRows * kTileK * 2;   // 12 KB per stage
    static constexpr int kStage = kX + kW;
    static constexpr int kPipe = kStages * kStage;      // 80 KB
    static constexpr int kOut = kTokPad * kTileRows * 4;  // 24 KB (aliases the pipeline)
    static_assert(kOut <= kPipe, "the output tile aliases the pipeline buffers");
    static constexpr int kBytes = kPipe;
};

// The tile's GEMM. rows_j[i] (shared) is the weight row of tile row i (-1: zero).
// On return out[t * kTileRows + i] (shared, aliasing the pipeline) holds the
// products for tokens t < kTokPad.
template <int MT>
__device__ void gu_tile(const WideLaunch& L, const __nv_bfloat16* w, const int* rows_j, unsigned char* sm,
                        float* out) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int d = L.d;
    const int nk = d / kTileK;
    // this thread's copies per stage: 3 weight chunks, 2 activation chunks
    const int wq = warp & 3, kh = warp >> 2;  // row tiles 3wq .. 3wq+2, K-steps 2kh, 2kh+1
    const __nv_bfloat16* wsrc[3];
    int wdst[3];
    bool wok[3];
#pragma unroll
    for (int i = 0; i < 3; ++i) {
        const int q = tid + kGuThreads * i;  // 768 chunks: row q / 8, chunk q % 8
        const int r = q >> 3, c = q & 7;
        const int j = rows_j[r];
        wok[i] = j >= 0;
        wsrc[i] = w + (size_t)(j >= 0 ? j : 0) * d + c * 8;
        wdst[i] = GuSmem::kX + swz(r, c, 128);
    }
    const __nv_bfloat16* xsrc[2];
    int xdst[2];
    bool xok[2];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const int q = tid + kGuThreads * i;  // 512 chunks: token q / 8, chunk q % 8
        const int t = q >> 3, c = q & 7;
        xok[i] = t < L.batch;
        xsrc[i] = L.x + (size_t)(t < L.batch ? t : 0) * d + c * 8;
        xdst[i] = swz(t, c, 128);
    }
    auto load = [&](int kst, int stage) {
        unsigned char* base = sm + stage * GuSmem::kStage;
        const int k0 = kst * kTileK;
#pragma unroll
        for (int i = 0; i < 3; ++i) cp16(base + wdst[i], wsrc[i] + k0, wok[i]);
#pragma unroll
        for (int i = 0; i < 2; ++i) cp16(base + xdst[i], xsrc[i] + k0, xok[i]);
    };

    float acc[MT][3][4];
#pragma unroll
    for (int a = 0; a < MT; ++a)
#pragma unroll
        for (int b = 0; b < 3; ++b)
#pragma unroll
            for (int e = 0; e < 4; ++e) acc[a][b][e] = 0.0f;

#pragma unroll
    for (int s = 0; s < kStages - 1; ++s) {
        if (s < nk) load(s, s);
        cp_commit();
    }
    for (int kst = 0; kst < nk; ++kst) {
        cp_wait<kStages - 2>();
        __syncthreads();  // the stage has landed for every thread; the oldest is free
        if (kst + kStages - 1 < nk) load(kst + kStages - 1, (kst + kStages - 1) % kStages);
        cp_commit();
        const uint32_t xs = smem_addr(sm + (kst % kStages) * GuSmem::kStage);
        const uint32_t ws = xs + GuSmem::kX;
#pragma unroll
        for (int k2 = 0; k2 < 2; ++k2) {
            const int kk = 2 * kh + k2;
            uint32_t af[MT][4];
#pragma unroll
            for (int mt = 0; mt < MT; ++mt) {
                // a0..a3: tokens 0-7 / 8-15 of the m-tile at k chunk 2kk / 2kk+1
                const int r = mt * 16 + (lane & 15);
                ldsm4(xs + swz(r, 2 * kk + (lane >> 4), 128), af[mt]);
            }
            uint32_t bf[4], b2a, b2b;
            {
                // row tiles 3w, 3w+1: (rows, k lo), (rows, k hi) for each
                const int r = wq * 24 + ((lane >> 4) << 3) + (lane & 7);
                ldsm4(ws + swz(r, 2 * kk + ((lane >> 3) & 1), 128), bf);
                const int r2 = wq * 24 + 16 + (lane & 7);
                ldsm2(ws + swz(r2, 2 * kk + ((lane >> 3) & 1), 128), b2a, b2b);
            }
#pragma unroll
            for (int mt = 0; mt < MT; ++mt) {
                mma16816(acc[mt][0], af[mt], bf[0], bf[1]);
                mma16816(acc[mt][1], af[mt], bf[2], bf[3]);
                mma16816(acc[mt][2], af[mt], b2a, b2b);
            }
        }
    }
    cp_wait<0>();
    __syncthreads();  // the pipeline buffers become the output tile
    // the second K half first, then the first half adds its own (fixed order)
    const int g = lane >> 2, t4 = lane & 3;
    for (int half = 1; half >= 0; --half) {
        if (kh == half) {
#pragma unroll
            for (int mt = 0; mt < MT; ++mt)
#pragma unroll
                for (int nt = 0; nt < 3; ++nt) {
                    const int col = wq * 24 + nt * 8 + 2 * t4;
                    const int tok = mt * 16 + g;
                    float* o0 = out + tok * kTileRows + col;
                    float* o1 = out + (tok + 8) * kTileRows + col;
                    if (half == 1) {
                        o0[0] = acc[mt][nt][0];
                        o0[1] = acc[mt][nt][1];
                        o1[0] = acc[mt][nt][2];
                        o1[1] = acc[mt][nt][3];
                    } else {
                        o0[0] = acc[mt][nt][0] + o0[0];
                        o0[1] = acc[mt][nt][1] + o0[1];
                        o1[0] = acc[mt][nt][2] + o1[0];
                        o1[1] = acc[mt][nt][3] + o1[1];
                    }
                }
        }
        __syncthreads();
    }
}

template <int MT>
__global__ void __launch_bounds__(kGuThreads) k_wide_gate(const WideLaunch L) {
    extern __shared__ __align__(128) unsigned char sm[];
    __shared__ int rows_j[kTileRows];
    pdl_wait();
    pdl_launch_dependents();
    const int p0 = blockIdx.x * kTileRows;
    const int tid = threadIdx.x;
    if (tid < kTileRows) rows_j[tid] = p0 + tid < L.n_rows ? row_of(L, p0 + tid) : -1;
    __syncthreads();
    float* out = reinterpret_cast<float*>(sm);
    gu_tile<MT>(L, L.wg, rows_j, sm, out);
    // g values, per-token gate bitmap bytes (and cleared both bytes) for the tile
    const int n_in = min(kTileRows, L.n_rows - p0);
    for (int q = tid; q < L.batch * kTileRows; q += kGuThreads) {
        const int t = q / kTileRows, i = q % kTileRows;
        if (i < n_in) L.gval[(size_t)t * L.n_rows + p0 + i] = out[t * kTileRows + i];
    }
    const int n_bytes = (n_in + 7) / 8;
    for (int q = tid; q < L.batch * n_bytes; q += kGuThreads) {
        const int t = q / n_bytes, b = q % n_bytes;
        unsigned bits = 0u;
        for (int r = 0; r < 8; ++r) {
            const int i = b * 8 + r;
            if (i < n_in && rows_j[i] >= 0 && out[t * kTileRows + i] > 0.0f) bits |= 1u << r;
        }
        L.gbits[(size_t)t * L.nbytes + p0 / 8 + b] = (uint8_t)bits;
        L.bbits[(size_t)t * L.nbytes + p0 / 8 + b] = 0;
    }
    for (int b = tid; b < n_bytes; b += kGuThreads) {
        unsigned u = 0u;
        for (int t = 0; t < L.batch; ++t)
            for (int r = 0; r < 8; ++r) {
                const int i = b * 8 + r;
                if (i < n_in && rows_j[i] >= 0 && out[t * kTileRows + i] > 0.0f) u |= 1u << r;
            }
        L.ugbits[p0 / 8 + b] = (uint8_t)u;
        L.ubits[p0 / 8 + b] = 0;
    }
}

template <int MT>
__global__ void __launch_bounds__(kGuThreads) k_wide_up(const WideLaunch L) {
    extern __shared__ __align__(128) unsigned char sm[];
    __shared__ int rows_j[kTileRows];
    __shared__ int pos[kTileRows];
    __shared__ int s_part[kGuThreads + 1];
    pdl_wait();
    pdl_launch_dependents();
    const int tid = threadIdx.x;
    const unsigned* ug = reinterpret_cast<const unsigned*>(L.ugbits);
    const BitScan bs = bit_scan<kGuThreads>(ug, L.n_rows, s_part);
    const int i0 = blockIdx.x * kTileRows;
    if (i0 >= bs.total) return;  // the union gate-active list is shorter
    const int n_in = min(kTileRows, bs.total - i0);
    if (tid < kTileRows) pos[tid] = -1;
    __syncthreads();
    bit_emit(ug, L.n_rows, bs, i0, i0 + n_in, pos);
    __syncthreads();
    if (tid < kTileRows) rows_j[tid] = pos[tid] >= 0 ? (L.rows ? L.rows[pos[tid]] : pos[tid]) : -1;
    __syncthreads();
    float* out = reinterpret_cast<float*>(sm);
    gu_tile<MT>(L, L.wu, rows_j, sm, out);
    // c = g u where both are positive (Eq. 2), split into bf16 hi + lo
    unsigned* bb = reinterpret_cast<unsigned*>(L.bbits);
    unsigned* ub = reinterpret_cast<unsigned*>(L.ubits);
    for (int q = tid; q < n_in * kTokPad; q += kGuThreads) {
        const int i = q / kTokPad, t = q % kTokPad;
        const int p = pos[i];
        float c = 0.0f;
        if (t < L.batch) {
            const float gv = L.gval[(size_t)t * L.n_rows + p];
            const float uv = out[t * kTileRows + i];
            if (gv > 0.0f && uv > 0.0f) {
                c = gv * uv;
                atomicOr(bb + (size_t)t * (L.nbytes / 4) + p / 32, 1u << (p % 32));
                atomicOr(ub + p / 32, 1u << (p % 32));
            }
        }
        const __nv_bfloat16 hi = __float2bfloat16_rn(c);
        L.c_hi[(size_t)p * kTokPad + t] = hi;
        L.c_lo[(size_t)p * kTokPad + t] = __float2bfloat16_rn(c - __bfloat162float(hi));
    }
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
                const int j = p >= 0 ? (L.rows ? L.rows[p] : p) : 0;
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

template <int MT>
cudaError_t run_t(const WideLaunch& L, cudaStream_t stream, bool pdl) {
    const int gu_grid = (L.n_rows + kTileRows - 1) / kTileRows;
    cudaError_t e = launch(k_wide_gate<MT>, gu_grid, kGuThreads, GuSmem::kBytes, stream, pdl, L);
    if (e == cudaSuccess) e = launch(k_wide_up<MT>, gu_grid, kGuThreads, GuSmem::kBytes, stream, true, L);
    if (e == cudaSuccess)
        e = launch(k_wide_down<MT>, (L.d / kDownCols) * L.ks, kDownThreads, DnSmem::kBytes, stream, true, L);
    if (e == cudaSuccess) {
        const int n = L.batch * L.d;
        e = launch(k_wide_reduce, (n + 255) / 256, 256, 0, stream, true, L);
    }
    return e;
}

template <int MT>
cudaError_t prepare_t() {
    cudaError_t e = cudaFuncSetAttribute(k_wide_gate<MT>, cudaFuncAttributeMaxDynamicSharedMemorySize, GuSmem::kBytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_wide_up<MT>, cudaFuncAttributeMaxDynamicSharedMemorySize, GuSmem::kBytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_wide_down<MT>, cudaFuncAttributeMaxDynamicSharedMemorySize, DnSmem::kBytes);
    return e;
}

}  // namespace

bool wide_supported(int wdtype, int d, int m, int batch) {
    return wdtype == 1 && batch > kMaxPass && batch <= kTokPad && d % kDownCols == 0 && m <= kScanWords * 32;
}

int wide_slices(int d, int num_sms) {
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
