// ts_api.cu -- the C ABI of libtsffn (declared in include/ts_ffn.h): handles,
// scratch arenas, argument validation, pass splitting, launch sequencing
// with programmatic dependent launch, active-set export and graph capture.
#include <nvtx3/nvToolsExt.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <new>
#include <vector>

#include "ts_ffn.h"
#include "ts_kernels.cuh"
#include "ts_predict.h"
#include "ts_wide.h"

using namespace tsffn;

namespace {

constexpr size_t kAlign = 256;
// rows of the next layer's W_gate each gate+up CTA prefetches into L2 (stack
// mode, passes of 4-8 tokens: the gathered down kernel issues them)
constexpr int kPrefetchRows = 32;

size_t align_up(size_t v) { return (v + kAlign - 1) / kAlign * kAlign; }
bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }
int elem_size(ts_dtype dt) { return dt == TS_BF16 ? 2 : 4; }  // fp32 / bf16 weights
// activations: bf16 for bf16 and INT4 weights, fp32 for fp32 weights
int act_size(ts_dtype dt) { return dt == TS_F32 ? 4 : 2; }
ts_dtype act_dtype(ts_dtype dt) { return dt == TS_F32 ? TS_F32 : TS_BF16; }
size_t weight_row_bytes(ts_dtype dt, int d) {
    return dt == TS_INT4 ? (size_t)d / 2 + (size_t)(d / 32) * 2 : (size_t)d * elem_size(dt);
}
int pow2_tokens(int nt) { return nt <= 1 ? 1 : nt <= 2 ? 2 : nt <= 4 ? 4 : 8; }

// Device facts needed to size grids; looked up at handle creation.
struct DeviceInfo {
    int device = 0;
    int num_sms = 1;
    int optin_smem = 48 * 1024;
};

ts_status device_info(DeviceInfo* di) {
    if (cudaGetDevice(&di->device) != cudaSuccess) return TS_ERR_CUDA;
    if (cudaDeviceGetAttribute(&di->num_sms, cudaDevAttrMultiProcessorCount, di->device) != cudaSuccess)
        return TS_ERR_CUDA;
    if (cudaDeviceGetAttribute(&di->optin_smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, di->device) !=
        cudaSuccess)
        return TS_ERR_CUDA;
    if (prepare_gate_up(di->optin_smem) != cudaSuccess || prepare_down() != cudaSuccess ||
        prepare_router() != cudaSuccess || prepare_wide() != cudaSuccess ||
        prepare_predict(di->optin_smem) != cudaSuccess)
        return TS_ERR_CUDA;
    return TS_OK;
}

// Carves sub-buffers out of one device allocation.
// One NVTX range per layer of the stack calls, so that a profiler's timeline
// shows the layers (header-only NVTX: with no tool attached the calls return
// at once). The ranges are host-side: inside a stream capture they mark the
// capture, not the graph's replays.
struct LayerRange {
    LayerRange(const char* what, int l) {
        char name[64];
        snprintf(name, sizeof name, "%s layer %d", what, l);
        nvtxRangePushA(name);
    }
    ~LayerRange() { nvtxRangePop(); }
    LayerRange(const LayerRange&) = delete;
    LayerRange& operator=(const LayerRange&) = delete;
};

// A handle's device scratch: blocks carved out of one allocation. Every block
// is followed by a guard zone of kGuardBytes filled with kGuardByte when the
// arena is allocated; check_arena reads the zones back, so a kernel that
// writes past the end of a scratch block is caught by the tests instead of
// silently corrupting the next block.
constexpr size_t kGuardBytes = kAlign;
constexpr unsigned char kGuardByte = 0xA5;

struct Arena {
    size_t bytes = 0;
    char* base = nullptr;
    std::vector<size_t> guards;  // offsets of the guard zones
    size_t take(size_t n) {
        const size_t off = bytes;
        bytes += align_up(n);
        guards.push_back(bytes);
        bytes += kGuardBytes;
        return off;
    }
    template <typename P>
    P* at(size_t off) const { return reinterpret_cast<P*>(base + off); }
};

ts_status alloc_arena(Arena* ar) {
    if (cudaMalloc(&ar->base, ar->bytes) != cudaSuccess) {
        cudaGetLastError();
        ar->base = nullptr;
        return TS_ERR_OOM;
    }
    bool ok = cudaMemset(ar->base, 0, ar->bytes) == cudaSuccess;
    for (size_t g : ar->guards) ok = ok && cudaMemset(ar->base + g, kGuardByte, kGuardBytes) == cudaSuccess;
    if (!ok) {
        cudaFree(ar->base);
        ar->base = nullptr;
        return TS_ERR_CUDA;
    }
    return TS_OK;
}

// Synchronise `stream` and compare every guard zone with its fill.
ts_status check_arena(const Arena& ar, cudaStream_t stream) {
    if (!ar.base) return TS_ERR_INVALID_ARG;
    if (cudaStreamSynchronize(stream) != cudaSuccess) return TS_ERR_CUDA;
    std::vector<unsigned char> buf(kGuardBytes);
    for (size_t g : ar.guards) {
        if (cudaMemcpy(buf.data(), ar.base + g, kGuardBytes, cudaMemcpyDeviceToHost) != cudaSuccess)
            return TS_ERR_CUDA;
        for (unsigned char b : buf)
            if (b != kGuardByte) return TS_ERR_SCRATCH;
    }
    return TS_OK;
}

// Scratch of the grouped kernels: per-expert c values and bitmaps, and the
// device status word.
struct Scratch {
    float* cval = nullptr;
    uint8_t* gbits = nullptr;
    uint8_t* bbits = nullptr;
    uint8_t* ubits = nullptr;
    uint8_t* ugbits = nullptr;
    unsigned* status = nullptr;
    float* partial = nullptr;  // [gate+up CTA][kAccMaxTokens][d]
};

}  // namespace

struct ts_ffn {
    int d = 0, m = 0, max_batch = 0;
    ts_dtype dt = TS_BF16;
    const void* wg = nullptr;
    const void* wu = nullptr;
    const void* wd = nullptr;
    DeviceInfo dev;
    int nbytes = 0;
    Arena arena;
    Scratch s;
    int grid[9] = {0};  // gate+up grid per pass width 1, 2, 4, 8
    // the last gate+up on this handle (read by ts_ffn_down and the exports)
    int last_batch = 0;
    const int32_t* last_rows = nullptr;
    int last_n_rows = 0;
    int test_stall = 0;  // ts_ffn_set_test_stall
    int pass_max = kMaxPass;  // tokens per pass (kAccMaxTokens for INT4 rows)
    // scratch of the wide kernels (batches of 9-64 tokens), when they apply
    bool wide = false;
    int wide_ks = 0;
    float* w_gval = nullptr;            // [max_batch][m]
    __nv_bfloat16* w_chi = nullptr;     // [m][64]
    __nv_bfloat16* w_clo = nullptr;     // [m][64]
    float* w_partial = nullptr;         // [ks][max_batch][d]
    __nv_bfloat16* w_x = nullptr;       // [max_batch][d] normalised activations (stack)
};

struct ts_moe {
    int d = 0, m = 0, E = 0, top_k = 0, max_batch = 0;
    ts_dtype dt = TS_BF16;
    const void* wr = nullptr;
    ExpertPtrs ex[kMaxExperts];
    DeviceInfo dev;
    int nbytes = 0;
    Arena arena;
    Scratch s;
    TokenRoute* route = nullptr;
    void* xbuf = nullptr;
    int grid[9] = {0};
    int last_batch = 0;
};

struct ts_predictor {
    int d = 0, r = 0, m = 0, max_batch = 0;
    ts_dtype dt = TS_BF16;
    const void* w1 = nullptr;  // [r][d]
    const void* w2 = nullptr;  // [m][r]
    DeviceInfo dev;
    Arena arena;
    float* hid = nullptr;      // [kPredMaxSplits][max_batch][r]
    unsigned* key = nullptr;   // [m]
    unsigned* hist = nullptr;  // [kPredHistParts][kPredHistBins]
};

struct ts_graph {
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    void* mem = nullptr;  // device memory the captured kernels read (fused stack: layer table, barrier)
};

extern "C" {

const char* ts_status_str(ts_status s) {
    switch (s) {
        case TS_OK: return "TS_OK";
        case TS_ERR_INVALID_ARG: return "TS_ERR_INVALID_ARG";
        case TS_ERR_CUDA: return "TS_ERR_CUDA";
        case TS_ERR_OOM: return "TS_ERR_OOM";
        case TS_ERR_BAD_INDEX: return "TS_ERR_BAD_INDEX";
        case TS_ERR_TIMEOUT: return "TS_ERR_TIMEOUT";
        case TS_ERR_UNSUPPORTED: return "TS_ERR_UNSUPPORTED";
        case TS_ERR_SCRATCH: return "TS_ERR_SCRATCH";
    }
    return "TS_ERR_UNKNOWN";
}

int ts_version(void) { return 100; }

ts_status ts_ffn_create(ts_ffn** out, int d, int m, ts_dtype wdtype, const void* w_gate,
                        const void* w_up, const void* w_down, int max_batch) {
    if (out == nullptr) return TS_ERR_INVALID_ARG;
    *out = nullptr;
    if (d < 1 || m < 1 || max_batch < 1 || max_batch > kMaxBatch) return TS_ERR_INVALID_ARG;
    if (wdtype != TS_F32 && wdtype != TS_BF16 && wdtype != TS_INT4) return TS_ERR_INVALID_ARG;
    if (!w_gate || !w_up || !w_down) return TS_ERR_INVALID_ARG;
    if (!aligned16(w_gate) || !aligned16(w_up) || !aligned16(w_down)) return TS_ERR_INVALID_ARG;
    if (wdtype == TS_INT4 ? d % 256 != 0 : ((size_t)d * elem_size(wdtype)) % 16 != 0) return TS_ERR_INVALID_ARG;
    if (m > (1 << 28) || (size_t)d * (size_t)m > ((size_t)1 << 40)) return TS_ERR_UNSUPPORTED;

    DeviceInfo dev;
    ts_status st = device_info(&dev);
    if (st != TS_OK) return st;
    const int pass_max = wdtype == TS_INT4 ? kAccMaxTokens : kMaxPass;  // INT4: passes of 1-2 tokens
    const int pass_cap = std::min(max_batch, pass_max);
    if (wdtype == TS_INT4) {
        if (!int4_supported(d, pass_cap, dev.optin_smem)) return TS_ERR_UNSUPPORTED;
    } else {
        int slots, slot_bytes, xs_stride;
        size_t smem;
        if (gate_up_config(wdtype, d, pass_cap, dev.optin_smem, &slots, &slot_bytes, &xs_stride, &smem) != 0)
            return TS_ERR_UNSUPPORTED;
    }

    ts_ffn* h = new (std::nothrow) ts_ffn();
    if (!h) return TS_ERR_OOM;
    h->d = d;
    h->m = m;
    h->max_batch = max_batch;
    h->dt = wdtype;
    h->wg = w_gate;
    h->wu = w_up;
    h->wd = w_down;
    h->dev = dev;
    h->pass_max = pass_max;
    h->nbytes = (m + 31) / 32 * 4;
    const int n_chunks = (m + kChunk - 1) / kChunk;
    for (int nt : {1, 2, 4, 8}) h->grid[nt] = std::max(1, std::min(dev.num_sms, n_chunks));
    const size_t o_cval = h->arena.take((size_t)kMaxPass * m * sizeof(float));
    const size_t o_p = h->arena.take((size_t)h->grid[kAccMaxTokens] * kAccMaxTokens * d * sizeof(float));
    const size_t o_g = h->arena.take((size_t)max_batch * h->nbytes);
    const size_t o_b = h->arena.take((size_t)max_batch * h->nbytes);
    const size_t o_u = h->arena.take((size_t)h->nbytes);
    const size_t o_ug = h->arena.take((size_t)h->nbytes);
    const size_t o_s = h->arena.take(sizeof(unsigned));
    h->wide = max_batch > kMaxPass && wide_supported(wdtype, d, m, max_batch);
    size_t o_wg = 0, o_whi = 0, o_wlo = 0, o_wp = 0, o_wx = 0;
    if (h->wide) {
        h->wide_ks = wide_slices(d, dev.num_sms);
        o_wg = h->arena.take((size_t)max_batch * m * sizeof(float));
        o_whi = h->arena.take((size_t)m * 64 * sizeof(__nv_bfloat16));
        o_wlo = h->arena.take((size_t)m * 64 * sizeof(__nv_bfloat16));
        o_wp = h->arena.take((size_t)h->wide_ks * max_batch * d * sizeof(float));
        o_wx = h->arena.take((size_t)max_batch * d * sizeof(__nv_bfloat16));
    }
    st = alloc_arena(&h->arena);
    if (st != TS_OK) {
        delete h;
        return st;
    }
    if (h->wide) {
        h->w_gval = h->arena.at<float>(o_wg);
        h->w_chi = h->arena.at<__nv_bfloat16>(o_whi);
        h->w_clo = h->arena.at<__nv_bfloat16>(o_wlo);
        h->w_partial = h->arena.at<float>(o_wp);
        h->w_x = h->arena.at<__nv_bfloat16>(o_wx);
    }
    h->s.cval = h->arena.at<float>(o_cval);
    h->s.gbits = h->arena.at<uint8_t>(o_g);
    h->s.bbits = h->arena.at<uint8_t>(o_b);
    h->s.ubits = h->arena.at<uint8_t>(o_u);
    h->s.ugbits = h->arena.at<uint8_t>(o_ug);
    h->s.status = h->arena.at<unsigned>(o_s);
    h->s.partial = h->arena.at<float>(o_p);
    *out = h;
    return TS_OK;
}

void ts_ffn_destroy(ts_ffn* h) {
    if (!h) return;
    if (h->arena.base) cudaFree(h->arena.base);
    delete h;
}

}  // extern "C"

namespace {

FfnLaunch ffn_launch(const ts_ffn* h, int batch, const int32_t* rows, int n_rows) {
    FfnLaunch a;
    memset(&a, 0, sizeof a);
    a.d = h->d;
    a.m = h->m;
    a.elem_bytes = h->dt == TS_INT4 ? 0 : elem_size(h->dt);
    a.row_bytes = (int)weight_row_bytes(h->dt, h->d);
    a.rows = rows;
    a.n_rows = rows ? n_rows : h->m;
    a.batch = batch;
    a.n_experts = 1;
    a.ex[0] = ExpertPtrs{h->wg, h->wu, h->wd};
    a.route = nullptr;
    a.top_k = 1;
    a.cval = h->s.cval;
    a.cval_tok_stride = h->m;
    a.gbits = h->s.gbits;
    a.bbits = h->s.bbits;
    a.bits_expert_stride = 0;
    a.nbytes = h->nbytes;
    a.ubits = h->s.ubits;
    a.ugbits = h->s.ugbits;
    a.status = h->s.status;
    a.partial = h->s.partial;
    a.partial_slots = kAccMaxTokens;
    a.test_stall = h->test_stall;
    return a;
}

ts_status cuda_status(cudaError_t e) { return e == cudaSuccess ? TS_OK : TS_ERR_CUDA; }

ts_status check_list(const ts_ffn* h, const int32_t* idx, int n) {
    if (idx != nullptr && (n < 0 || n > h->m)) return TS_ERR_INVALID_ARG;
    return TS_OK;
}

// gate+up (and down) for tokens tok0 .. tok0+nt-1 of the call.
ts_status run_pass(ts_ffn* h, FfnLaunch a, int tok0, int nt, cudaStream_t stream, bool gate_up,
                   bool down) {
    a.tok0 = tok0;
    a.nt = nt;
    a.bits_tok_base = tok0;
    const int w = pow2_tokens(nt);
    a.partial_ctas = h->grid[w];
    if (gate_up) {
        ts_status st = cuda_status(launch_gate_up(a, h->dt, w, h->grid[w], stream, true));
        if (st != TS_OK) return st;
    }
    if (down)
        return cuda_status(w <= kAccMaxTokens ? launch_down_reduce(a, w, stream, true)
                                              : launch_down(a, h->dt, w, stream, true));
    return TS_OK;
}

// The whole batch in one wide pass (9-64 tokens, bf16 rows).
bool use_wide(const ts_ffn* h, int batch) { return h->wide && wide_supported(h->dt, h->d, h->m, batch); }

WideLaunch wide_launch(const ts_ffn* h, int batch, const int32_t* rows, int n_rows) {
    WideLaunch L;
    memset(&L, 0, sizeof L);
    L.d = h->d;
    L.m = h->m;
    L.rows = rows;
    L.n_rows = rows ? n_rows : h->m;
    L.batch = batch;
    L.wg = static_cast<const __nv_bfloat16*>(h->wg);
    L.wu = static_cast<const __nv_bfloat16*>(h->wu);
    L.wd = static_cast<const __nv_bfloat16*>(h->wd);
    L.gval = h->w_gval;
    L.c_hi = h->w_chi;
    L.c_lo = h->w_clo;
    L.partial = h->w_partial;
    L.ks = h->wide_ks;
    L.gbits = h->s.gbits;
    L.bbits = h->s.bbits;
    L.ubits = h->s.ubits;
    L.ugbits = h->s.ugbits;
    L.nbytes = h->nbytes;
    L.status = h->s.status;
    return L;
}

void remember(ts_ffn* h, int batch, const int32_t* rows, int n_rows) {
    h->last_batch = batch;
    h->last_rows = rows;
    h->last_n_rows = rows ? n_rows : h->m;
}

// Decode bitmap bytes of the row space into ascending neuron ids.
int decode_bits(const uint8_t* bits, int n_rows, const std::vector<int32_t>& rows, int32_t* out) {
    int n = 0;
    for (int p = 0; p < n_rows; ++p)
        if ((bits[p >> 3] >> (p & 7)) & 1u) {
            if (out) out[n] = rows.empty() ? p : rows[p];
            ++n;
        }
    return n;
}

// Host copies of per-token bitmaps (token >= 0) or their union over `tokens`.
ts_status fetch_active(cudaStream_t stream, const uint8_t* gbits_dev, const uint8_t* bbits_dev,
                       int nbytes, int n_rows, const int32_t* rows_dev, int token_first,
                       int n_tokens, int32_t* gate_idx, int* n_gate, int32_t* both_idx, int* n_both) {
    if (cudaStreamSynchronize(stream) != cudaSuccess) return TS_ERR_CUDA;
    std::vector<uint8_t> g((size_t)n_tokens * nbytes), b((size_t)n_tokens * nbytes);
    if (n_tokens > 0) {
        if (cudaMemcpy(g.data(), gbits_dev + (size_t)token_first * nbytes, g.size(),
                       cudaMemcpyDeviceToHost) != cudaSuccess ||
            cudaMemcpy(b.data(), bbits_dev + (size_t)token_first * nbytes, b.size(),
                       cudaMemcpyDeviceToHost) != cudaSuccess)
            return TS_ERR_CUDA;
    }
    std::vector<uint8_t> gu(nbytes, 0), bu(nbytes, 0);
    for (int t = 0; t < n_tokens; ++t)
        for (int i = 0; i < nbytes; ++i) {
            gu[i] |= g[(size_t)t * nbytes + i];
            bu[i] |= b[(size_t)t * nbytes + i];
        }
    std::vector<int32_t> rows;
    if (rows_dev != nullptr && n_rows > 0) {
        rows.resize(n_rows);
        if (cudaMemcpy(rows.data(), rows_dev, n_rows * sizeof(int32_t), cudaMemcpyDeviceToHost) !=
            cudaSuccess)
            return TS_ERR_CUDA;
    }
    const int ng = decode_bits(gu.data(), n_rows, rows, gate_idx);
    const int nb = decode_bits(bu.data(), n_rows, rows, both_idx);
    if (n_gate) *n_gate = ng;
    if (n_both) *n_both = nb;
    return TS_OK;
}

ts_status read_status(unsigned* status_dev, cudaStream_t stream) {
    unsigned v = 0;
    if (cudaStreamSynchronize(stream) != cudaSuccess) return TS_ERR_CUDA;
    if (cudaMemcpy(&v, status_dev, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess) return TS_ERR_CUDA;
    if (cudaMemset(status_dev, 0, sizeof v) != cudaSuccess) return TS_ERR_CUDA;
    if (v & kStatusTimeout) return TS_ERR_TIMEOUT;
    return (v & kStatusBadIndex) ? TS_ERR_BAD_INDEX : TS_OK;
}

// One layer of the residual stack: h += FFN(rmsnorm(h)) over the layer's
// rows (all, or the list). `next` is the following layer when it runs dense
// (its first W_gate rows are then prefetched into L2), else nullptr.
ts_status stack_layer(ts_ffn* h, const ts_ffn* next, float* hres, int batch, const int32_t* rows, int nr,
                      cudaStream_t stream, bool rows_ready, bool h_ready = false, bool trigger_early = false) {
    if (use_wide(h, batch)) {
        WideLaunch L = wide_launch(h, batch, rows, nr);
        L.x = h->w_x;
        L.h = hres;
        L.residual_out = 1;
        ts_status st = cuda_status(launch_wide_norm(L, hres, h->w_x, stream, true));
        if (st == TS_OK) st = cuda_status(launch_wide(L, stream, true));
        if (st != TS_OK) return st;
        remember(h, batch, rows, nr);
        return TS_OK;
    }
    FfnLaunch a = ffn_launch(h, batch, rows, nr);
    a.h = hres;
    a.norm_from_h = 1;
    a.residual_out = 1;
    a.rows_ready = rows != nullptr && rows_ready ? 1 : 0;
    a.h_ready = h_ready ? 1 : 0;
    a.trigger_early = trigger_early ? 1 : 0;
    if (next != nullptr && batch <= kMaxPass && h->dt != TS_INT4) {
        a.next_wg = next->wg;
        a.next_n_rows = next->m;
        a.next_grid = next->grid[pow2_tokens(std::min(kMaxPass, batch))];
        a.prefetch_rows = kPrefetchRows;
    }
    for (int t0 = 0; t0 < batch; t0 += h->pass_max) {
        ts_status st = run_pass(h, a, t0, std::min(h->pass_max, batch - t0), stream, true, true);
        if (st != TS_OK) return st;
    }
    remember(h, batch, rows, nr);
    return TS_OK;
}

}  // namespace

extern "C" {

ts_status ts_ffn_forward(ts_ffn* h, const void* x, int batch, float* y, cudaStream_t stream,
                         const int32_t* active_idx, int n_active) {
    if (!h || batch < 0 || batch > h->max_batch) return TS_ERR_INVALID_ARG;
    if (batch == 0) return TS_OK;
    if (!x || !y) return TS_ERR_INVALID_ARG;
    ts_status st = check_list(h, active_idx, n_active);
    if (st != TS_OK) return st;
    if (use_wide(h, batch)) {
        WideLaunch L = wide_launch(h, batch, active_idx, n_active);
        L.x = static_cast<const __nv_bfloat16*>(x);
        L.y = y;
        st = cuda_status(launch_wide(L, stream, true));
        if (st == TS_OK) remember(h, batch, active_idx, n_active);
        return st;
    }
    FfnLaunch a = ffn_launch(h, batch, active_idx, n_active);
    a.x = x;
    a.y = y;
    for (int t0 = 0; t0 < batch; t0 += h->pass_max) {
        st = run_pass(h, a, t0, std::min(h->pass_max, batch - t0), stream, true, true);
        if (st != TS_OK) return st;
    }
    remember(h, batch, active_idx, n_active);
    return TS_OK;
}

ts_status ts_ffn_forward_topk(ts_ffn* h, const void* x, int batch, float* y, cudaStream_t stream, int keep) {
    if (!h || batch < 0 || batch > h->max_batch || keep < 0 || keep > h->m) return TS_ERR_INVALID_ARG;
    if (h->dt == TS_INT4) return TS_ERR_UNSUPPORTED;
    if (batch == 0) return TS_OK;
    if (!x || !y) return TS_ERR_INVALID_ARG;
    FfnLaunch a = ffn_launch(h, batch, nullptr, 0);
    a.x = x;
    a.y = y;
    for (int t0 = 0; t0 < batch; t0 += kMaxPass) {
        // the down projection runs after the mask: passes of 1-2 tokens take
        // the row kernel without its per-CTA down partial (a null partial
        // buffer), then the mask, then the gathered down kernel
        const int nt = std::min(kMaxPass, batch - t0);
        const int w = nt <= kAccMaxTokens ? pow2_tokens(nt) : std::max(4, pow2_tokens(nt));
        a.tok0 = t0;
        a.nt = nt;
        a.bits_tok_base = t0;
        a.partial = w <= kAccMaxTokens ? nullptr : h->s.partial;
        a.partial_ctas = h->grid[w];
        ts_status st = cuda_status(launch_gate_up(a, h->dt, w, h->grid[w], stream, true));
        if (st == TS_OK) st = cuda_status(launch_topk(a, keep, stream));
        if (st == TS_OK) st = cuda_status(launch_down(a, h->dt, w, stream, true));
        if (st != TS_OK) return st;
    }
    remember(h, batch, nullptr, 0);
    return TS_OK;
}

ts_status ts_ffn_gate_up(ts_ffn* h, const void* x, int batch, cudaStream_t stream,
                         const int32_t* active_idx, int n_active) {
    if (!h || batch < 0 || batch > h->max_batch) return TS_ERR_INVALID_ARG;
    if (batch > h->pass_max) return TS_ERR_UNSUPPORTED;
    if (batch == 0) return TS_OK;
    if (!x) return TS_ERR_INVALID_ARG;
    ts_status st = check_list(h, active_idx, n_active);
    if (st != TS_OK) return st;
    FfnLaunch a = ffn_launch(h, batch, active_idx, n_active);
    a.x = x;
    st = run_pass(h, a, 0, batch, stream, true, false);
    if (st == TS_OK) remember(h, batch, active_idx, n_active);
    return st;
}

ts_status ts_ffn_down(ts_ffn* h, int batch, float* y, cudaStream_t stream) {
    if (!h || batch < 0 || batch > h->pass_max) return TS_ERR_INVALID_ARG;
    if (batch == 0) return TS_OK;
    if (!y || batch != h->last_batch) return TS_ERR_INVALID_ARG;
    FfnLaunch a = ffn_launch(h, batch, h->last_rows, h->last_n_rows);
    a.y = y;
    return run_pass(h, a, 0, batch, stream, false, true);
}

ts_status ts_stack_forward(ts_ffn* const* layers, int n_layers, float* hres, int batch,
                           cudaStream_t stream, const int32_t* const* active_idx,
                           const int* n_active) {
    if (!layers || n_layers < 0 || !hres || batch < 0) return TS_ERR_INVALID_ARG;
    if (batch == 0 || n_layers == 0) return TS_OK;
    for (int l = 0; l < n_layers; ++l) {
        const ts_ffn* h = layers[l];
        if (!h || h->d != layers[0]->d || h->dt != layers[0]->dt || batch > h->max_batch)
            return TS_ERR_INVALID_ARG;
        const int32_t* rows = active_idx ? active_idx[l] : nullptr;
        if (rows && !n_active) return TS_ERR_INVALID_ARG;
        ts_status st = check_list(h, rows, rows ? n_active[l] : 0);
        if (st != TS_OK) return st;
    }
    for (int l = 0; l < n_layers; ++l) {
        const int32_t* rows = active_idx ? active_idx[l] : nullptr;
        const bool next_dense = l + 1 < n_layers && !(active_idx && active_idx[l + 1]);
        // a caller's list is in memory before the stack starts; from the
        // second layer on, every kernel before the launch has finished with
        // the first layer's wait, so the list may be read before waiting
        LayerRange range("ffn stack", l);
        ts_status st = stack_layer(layers[l], next_dense ? layers[l + 1] : nullptr, hres, batch, rows,
                                   rows ? n_active[l] : 0, stream, l > 0, false, l + 1 < n_layers);
        if (st != TS_OK) return st;
    }
    return TS_OK;
}

ts_status ts_ffn_get_active(ts_ffn* h, cudaStream_t stream, int token, int32_t* gate_idx,
                            int* n_gate, int32_t* both_idx, int* n_both) {
    if (!h || token < -1 || token >= std::max(h->last_batch, 0)) return TS_ERR_INVALID_ARG;
    if (h->last_batch == 0) return TS_ERR_INVALID_ARG;
    const int first = token < 0 ? 0 : token;
    const int n = token < 0 ? h->last_batch : 1;
    return fetch_active(stream, h->s.gbits, h->s.bbits, h->nbytes, h->last_n_rows, h->last_rows,
                        first, n, gate_idx, n_gate, both_idx, n_both);
}

ts_status ts_ffn_get_error(ts_ffn* h, cudaStream_t stream) {
    if (!h) return TS_ERR_INVALID_ARG;
    return read_status(h->s.status, stream);
}

ts_status ts_ffn_check_scratch(ts_ffn* h, cudaStream_t stream) {
    if (!h) return TS_ERR_INVALID_ARG;
    return check_arena(h->arena, stream);
}

ts_status ts_ffn_poke_guard(ts_ffn* h, int i) {
    if (!h || !h->arena.base || i < 0 || (size_t)i >= h->arena.guards.size()) return TS_ERR_INVALID_ARG;
    const unsigned char v = (unsigned char)~kGuardByte;
    return cudaMemcpy(h->arena.base + h->arena.guards[(size_t)i], &v, 1, cudaMemcpyHostToDevice) == cudaSuccess
               ? TS_OK
               : TS_ERR_CUDA;
}

ts_status ts_ffn_set_test_stall(ts_ffn* h, int on) {
    if (!h) return TS_ERR_INVALID_ARG;
    h->test_stall = on ? 1 : 0;
    return TS_OK;
}

// ---------------------------------------------------------------------------
// MoE
// ---------------------------------------------------------------------------
ts_status ts_moe_create(ts_moe** out, int d, int n_experts, int top_k, ts_dtype wdtype,
                        const void* w_router, ts_ffn* const* experts, int max_batch) {
    if (out == nullptr) return TS_ERR_INVALID_ARG;
    *out = nullptr;
    if (d < 1 || n_experts < 1 || n_experts > kMaxExperts) return TS_ERR_INVALID_ARG;
    if (top_k < 1 || top_k > std::min(kMaxTopK, n_experts)) return TS_ERR_INVALID_ARG;
    if (max_batch < 1 || max_batch > kMaxMoeBatch) return TS_ERR_INVALID_ARG;
    if (wdtype != TS_F32 && wdtype != TS_BF16 && wdtype != TS_INT4) return TS_ERR_INVALID_ARG;
    if (!w_router || !aligned16(w_router) || !experts) return TS_ERR_INVALID_ARG;
    if (wdtype == TS_INT4 && max_batch > kAccMaxTokens) return TS_ERR_UNSUPPORTED;
    if (d > kRouterMaxD) return TS_ERR_UNSUPPORTED;
    for (int e = 0; e < n_experts; ++e) {
        const ts_ffn* x = experts[e];
        if (!x || x->d != d || x->dt != wdtype || x->m != experts[0]->m) return TS_ERR_INVALID_ARG;
    }
    DeviceInfo dev;
    ts_status st = device_info(&dev);
    if (st != TS_OK) return st;
    if (wdtype == TS_INT4) {
        if (!int4_supported(d, max_batch, dev.optin_smem)) return TS_ERR_UNSUPPORTED;
    } else {
        int slots, slot_bytes, xs_stride;
        size_t smem;
        if (gate_up_config(wdtype, d, max_batch, dev.optin_smem, &slots, &slot_bytes, &xs_stride, &smem) != 0)
            return TS_ERR_UNSUPPORTED;
    }

    ts_moe* h = new (std::nothrow) ts_moe();
    if (!h) return TS_ERR_OOM;
    h->d = d;
    h->m = experts[0]->m;
    h->E = n_experts;
    h->top_k = top_k;
    h->max_batch = max_batch;
    h->dt = wdtype;
    h->wr = w_router;
    for (int e = 0; e < n_experts; ++e) h->ex[e] = ExpertPtrs{experts[e]->wg, experts[e]->wu, experts[e]->wd};
    h->dev = dev;
    h->nbytes = (h->m + 31) / 32 * 4;
    const int m = h->m, E = n_experts;
    const int n_chunks = (m + kChunk - 1) / kChunk;
    for (int nt : {1, 2, 4, 8})
        h->grid[nt] = std::max(1, std::min(dev.num_sms, std::min(E, nt * top_k) * n_chunks));
    const size_t o_cval = h->arena.take((size_t)E * kMaxPass * m * sizeof(float));
    const size_t o_p = h->arena.take((size_t)h->grid[kAccMaxTokens] * kAccMaxTokens * d * sizeof(float));
    const size_t o_g = h->arena.take((size_t)E * kMaxPass * h->nbytes);
    const size_t o_b = h->arena.take((size_t)E * kMaxPass * h->nbytes);
    const size_t o_u = h->arena.take((size_t)E * h->nbytes);
    const size_t o_ug = h->arena.take((size_t)E * h->nbytes);
    const size_t o_s = h->arena.take(sizeof(unsigned));
    const size_t o_r = h->arena.take((size_t)max_batch * sizeof(TokenRoute));
    const size_t o_x = h->arena.take((size_t)max_batch * d * act_size(wdtype));
    st = alloc_arena(&h->arena);
    if (st != TS_OK) {
        delete h;
        return st;
    }
    h->s.cval = h->arena.at<float>(o_cval);
    h->s.gbits = h->arena.at<uint8_t>(o_g);
    h->s.bbits = h->arena.at<uint8_t>(o_b);
    h->s.ubits = h->arena.at<uint8_t>(o_u);
    h->s.ugbits = h->arena.at<uint8_t>(o_ug);
    h->s.status = h->arena.at<unsigned>(o_s);
    h->route = h->arena.at<TokenRoute>(o_r);
    h->xbuf = h->arena.at<void>(o_x);
    h->s.partial = h->arena.at<float>(o_p);
    *out = h;
    return TS_OK;
}

void ts_moe_destroy(ts_moe* h) {
    if (!h) return;
    if (h->arena.base) cudaFree(h->arena.base);
    delete h;
}

}  // extern "C"

namespace {

// router -> grouped gate+up -> grouped down for one MoE layer.
ts_status moe_layer(ts_moe* h, const void* x, float* hres, int batch, float* y, cudaStream_t stream) {
    RouterLaunch r;
    memset(&r, 0, sizeof r);
    r.d = h->d;
    r.n_experts = h->E;
    r.top_k = h->top_k;
    r.batch = batch;
    r.x = hres ? nullptr : x;
    r.h = hres;
    r.xbuf = h->xbuf;
    r.wr = h->wr;
    r.route = h->route;
    // the router and its normalised activations use the activation type
    ts_status st = cuda_status(launch_router(r, act_dtype(h->dt), stream, true));
    if (st != TS_OK) return st;

    FfnLaunch a;
    memset(&a, 0, sizeof a);
    a.d = h->d;
    a.m = h->m;
    a.elem_bytes = h->dt == TS_INT4 ? 0 : elem_size(h->dt);
    a.row_bytes = (int)weight_row_bytes(h->dt, h->d);
    a.n_rows = h->m;
    a.rows = nullptr;
    a.batch = batch;
    a.tok0 = 0;
    a.nt = batch;
    a.x = hres ? h->xbuf : x;
    a.h = hres;
    a.y = y;
    a.norm_from_h = 0;
    a.residual_out = hres ? 1 : 0;
    a.n_experts = h->E;
    for (int e = 0; e < h->E; ++e) a.ex[e] = h->ex[e];
    a.route = h->route;
    a.top_k = h->top_k;
    a.cval = h->s.cval;
    a.cval_tok_stride = h->m;
    a.gbits = h->s.gbits;
    a.bbits = h->s.bbits;
    a.bits_expert_stride = (long long)kMaxPass * h->nbytes;
    a.bits_tok_base = 0;
    a.nbytes = h->nbytes;
    a.ubits = h->s.ubits;
    a.ugbits = h->s.ugbits;
    a.status = h->s.status;
    const int w = pow2_tokens(batch);
    a.partial = h->s.partial;
    a.partial_slots = kAccMaxTokens;
    a.partial_ctas = h->grid[w];
    st = cuda_status(launch_gate_up(a, h->dt, w, h->grid[w], stream, true));
    if (st != TS_OK) return st;
    return cuda_status(w <= kAccMaxTokens ? launch_down_reduce(a, w, stream, true)
                                          : launch_down(a, h->dt, w, stream, true));
}

}  // namespace

extern "C" {

ts_status ts_moe_forward(ts_moe* h, const void* x, int batch, float* y, cudaStream_t stream) {
    if (!h || batch < 0 || batch > h->max_batch) return TS_ERR_INVALID_ARG;
    if (batch == 0) return TS_OK;
    if (!x || !y) return TS_ERR_INVALID_ARG;
    ts_status st = moe_layer(h, x, nullptr, batch, y, stream);
    if (st == TS_OK) h->last_batch = batch;
    return st;
}

ts_status ts_moe_stack_forward(ts_moe* const* layers, int n_layers, float* hres, int batch,
                               cudaStream_t stream) {
    if (!layers || n_layers < 0 || !hres || batch < 0) return TS_ERR_INVALID_ARG;
    if (batch == 0 || n_layers == 0) return TS_OK;
    for (int l = 0; l < n_layers; ++l) {
        const ts_moe* h = layers[l];
        if (!h || h->d != layers[0]->d || h->dt != layers[0]->dt || batch > h->max_batch)
            return TS_ERR_INVALID_ARG;
    }
    for (int l = 0; l < n_layers; ++l) {
        LayerRange range("moe stack", l);
        ts_status st = moe_layer(layers[l], nullptr, hres, batch, nullptr, stream);
        if (st != TS_OK) return st;
        layers[l]->last_batch = batch;
    }
    return TS_OK;
}

ts_status ts_moe_get_routing(ts_moe* h, cudaStream_t stream, int32_t* sel, float* w) {
    if (!h || h->last_batch == 0) return TS_ERR_INVALID_ARG;
    if (cudaStreamSynchronize(stream) != cudaSuccess) return TS_ERR_CUDA;
    std::vector<TokenRoute> r(h->last_batch);
    if (cudaMemcpy(r.data(), h->route, r.size() * sizeof(TokenRoute), cudaMemcpyDeviceToHost) !=
        cudaSuccess)
        return TS_ERR_CUDA;
    for (int t = 0; t < h->last_batch; ++t)
        for (int k = 0; k < h->top_k; ++k) {
            if (sel) sel[t * h->top_k + k] = r[t].sel[k];
            if (w) w[t * h->top_k + k] = r[t].w[k];
        }
    return TS_OK;
}

ts_status ts_moe_get_active(ts_moe* h, cudaStream_t stream, int expert, int token, int32_t* gate_idx,
                            int* n_gate, int32_t* both_idx, int* n_both) {
    if (!h || h->last_batch == 0 || expert < 0 || expert >= h->E) return TS_ERR_INVALID_ARG;
    if (token < -1 || token >= h->last_batch) return TS_ERR_INVALID_ARG;
    std::vector<int32_t> sel((size_t)h->last_batch * h->top_k);
    ts_status st = ts_moe_get_routing(h, stream, sel.data(), nullptr);
    if (st != TS_OK) return st;
    // local token index of each routed token, in token order
    std::vector<int> toks;
    for (int t = 0; t < h->last_batch; ++t)
        for (int k = 0; k < h->top_k; ++k)
            if (sel[(size_t)t * h->top_k + k] == expert) toks.push_back(t);
    const uint8_t* gb = h->s.gbits + (size_t)expert * kMaxPass * h->nbytes;
    const uint8_t* bb = h->s.bbits + (size_t)expert * kMaxPass * h->nbytes;
    if (token < 0)
        return fetch_active(stream, gb, bb, h->nbytes, h->m, nullptr, 0, (int)toks.size(), gate_idx,
                            n_gate, both_idx, n_both);
    const auto it = std::find(toks.begin(), toks.end(), token);
    if (it == toks.end()) {  // token not routed to this expert: nothing active
        if (n_gate) *n_gate = 0;
        if (n_both) *n_both = 0;
        return TS_OK;
    }
    return fetch_active(stream, gb, bb, h->nbytes, h->m, nullptr, (int)(it - toks.begin()), 1,
                        gate_idx, n_gate, both_idx, n_both);
}

ts_status ts_moe_get_error(ts_moe* h, cudaStream_t stream) {
    if (!h) return TS_ERR_INVALID_ARG;
    return read_status(h->s.status, stream);
}

ts_status ts_moe_check_scratch(ts_moe* h, cudaStream_t stream) {
    if (!h) return TS_ERR_INVALID_ARG;
    return check_arena(h->arena, stream);
}

// ---------------------------------------------------------------------------
// graphs
// ---------------------------------------------------------------------------
}  // extern "C"

extern "C" {

ts_status ts_predictor_create(ts_predictor** out, int d, int r, int m, ts_dtype dtype, const void* w1,
                              const void* w2, int max_batch) {
    if (out == nullptr) return TS_ERR_INVALID_ARG;
    *out = nullptr;
    if (d < 1 || r < 1 || m < 1 || max_batch < 1) return TS_ERR_INVALID_ARG;
    if (dtype != TS_F32 && dtype != TS_BF16) return TS_ERR_INVALID_ARG;
    if (!w1 || !w2 || !aligned16(w1) || !aligned16(w2)) return TS_ERR_INVALID_ARG;
    if (max_batch > kPredMaxBatch || m > (1 << 28)) return TS_ERR_UNSUPPORTED;
    DeviceInfo dev;
    ts_status st = device_info(&dev);
    if (st != TS_OK) return st;
    if (!predict_supported(elem_size(dtype), d, r, max_batch, dev.optin_smem)) return TS_ERR_UNSUPPORTED;
    ts_predictor* p = new (std::nothrow) ts_predictor();
    if (!p) return TS_ERR_OOM;
    p->d = d;
    p->r = r;
    p->m = m;
    p->max_batch = max_batch;
    p->dt = dtype;
    p->w1 = w1;
    p->w2 = w2;
    p->dev = dev;
    const size_t o_h = p->arena.take((size_t)kPredMaxSplits * max_batch * r * sizeof(float));
    const size_t o_k = p->arena.take((size_t)m * sizeof(unsigned));
    const size_t o_b = p->arena.take((size_t)kPredHistParts * kPredHistBins * sizeof(unsigned));
    st = alloc_arena(&p->arena);
    if (st != TS_OK) {
        delete p;
        return st;
    }
    p->hid = p->arena.at<float>(o_h);
    p->key = p->arena.at<unsigned>(o_k);
    p->hist = p->arena.at<unsigned>(o_b);
    *out = p;
    return TS_OK;
}

void ts_predictor_destroy(ts_predictor* p) {
    if (!p) return;
    if (p->arena.base) cudaFree(p->arena.base);
    delete p;
}

ts_status ts_predictor_check_scratch(ts_predictor* p, cudaStream_t stream) {
    if (!p) return TS_ERR_INVALID_ARG;
    return check_arena(p->arena, stream);
}

}  // extern "C"

namespace {

PredictLaunch predict_launch(const ts_predictor* p, int batch, int K, int32_t* list, float* scores) {
    PredictLaunch q;
    memset(&q, 0, sizeof q);
    q.d = p->d;
    q.r = p->r;
    q.m = p->m;
    q.batch = batch;
    q.w1 = p->w1;
    q.w2 = p->w2;
    q.hid = p->hid;
    q.key = p->key;
    q.hist = p->hist;
    q.scores = scores;
    q.K = K;
    q.list = list;
    predict_geometry(&q, elem_size(p->dt), p->dev.num_sms);
    return q;
}

}  // namespace

extern "C" {

ts_status ts_predict(ts_predictor* p, const void* x, int batch, int K, int32_t* list, float* scores,
                     cudaStream_t stream) {
    if (!p || batch < 0 || batch > p->max_batch || K < 0 || K > p->m) return TS_ERR_INVALID_ARG;
    if (batch == 0 || K == 0) return TS_OK;
    if (!x || !list || ((uintptr_t)x & (act_size(p->dt) - 1)) != 0 || ((uintptr_t)list & 3u) != 0)
        return TS_ERR_INVALID_ARG;
    PredictLaunch q = predict_launch(p, batch, K, list, scores);
    q.x = x;
    return cuda_status(launch_predict(q, elem_size(p->dt), stream, true));
}

ts_status ts_stack_forward_predicted(ts_ffn* const* layers, ts_predictor* const* preds, int n_layers,
                                     float* hres, int batch, const int* K, int32_t* const* lists,
                                     cudaStream_t stream) {
    if (!layers || !preds || n_layers < 0 || !hres || batch < 0) return TS_ERR_INVALID_ARG;
    if (batch == 0 || n_layers == 0) return TS_OK;
    if (!K || !lists) return TS_ERR_INVALID_ARG;
    for (int l = 0; l < n_layers; ++l) {
        const ts_ffn* h = layers[l];
        const ts_predictor* p = preds[l];
        if (!h || !p || h->d != layers[0]->d || h->dt != layers[0]->dt || batch > h->max_batch)
            return TS_ERR_INVALID_ARG;
        if (p->d != h->d || p->m != h->m || p->dt != act_dtype(h->dt) || batch > p->max_batch)
            return TS_ERR_INVALID_ARG;
        if (K[l] < 0 || K[l] > h->m || !lists[l] || ((uintptr_t)lists[l] & 3u) != 0) return TS_ERR_INVALID_ARG;
    }
    for (int l = 0; l < n_layers; ++l) {
        ts_ffn* h = layers[l];
        if (K[l] == 0) {  // an empty list: the layer adds nothing
            remember(h, batch, lists[l], 0);
            continue;
        }
        LayerRange range("predicted stack", l);
        PredictLaunch q = predict_launch(preds[l], batch, K[l], lists[l], nullptr);
        q.h = hres;
        ts_status st = cuda_status(launch_predict(q, elem_size(preds[l]->dt), stream, true));
        // the predictor's three kernels ran after the last writer of h
        // the reduction lets the next layer's predictor kernels be scheduled
        // before their wait, as it does for the next gate+up kernel
        if (st == TS_OK) st = stack_layer(h, nullptr, hres, batch, lists[l], K[l], stream, false, true, l + 1 < n_layers);
        if (st != TS_OK) return st;
    }
    return TS_OK;
}

}  // extern "C"

namespace {

template <typename F>
ts_status capture(ts_graph** out, F&& body) {
    if (!out) return TS_ERR_INVALID_ARG;
    *out = nullptr;
    cudaStream_t s;
    if (cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking) != cudaSuccess) return TS_ERR_CUDA;
    if (cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
        cudaStreamDestroy(s);
        return TS_ERR_CUDA;
    }
    ts_status st = body(s);
    cudaGraph_t g = nullptr;
    const cudaError_t ec = cudaStreamEndCapture(s, &g);
    cudaStreamDestroy(s);
    if (st != TS_OK || ec != cudaSuccess) {
        if (g) cudaGraphDestroy(g);
        return st != TS_OK ? st : TS_ERR_CUDA;
    }
    ts_graph* gr = new (std::nothrow) ts_graph();
    if (!gr) {
        cudaGraphDestroy(g);
        return TS_ERR_OOM;
    }
    gr->graph = g;
    if (cudaGraphInstantiate(&gr->exec, g, 0) != cudaSuccess) {
        cudaGraphDestroy(g);
        delete gr;
        return TS_ERR_CUDA;
    }
    *out = gr;
    return TS_OK;
}

}  // namespace

extern "C" {

ts_status ts_graph_capture_stack(ts_graph** out, ts_ffn* const* layers, int n_layers, float* h,
                                 int batch, const int32_t* const* active_idx, const int* n_active) {
    return capture(out, [&](cudaStream_t s) {
        return ts_stack_forward(layers, n_layers, h, batch, s, active_idx, n_active);
    });
}

ts_status ts_graph_capture_moe_stack(ts_graph** out, ts_moe* const* layers, int n_layers, float* h,
                                     int batch) {
    return capture(out, [&](cudaStream_t s) { return ts_moe_stack_forward(layers, n_layers, h, batch, s); });
}

ts_status ts_graph_capture_stack_predicted(ts_graph** out, ts_ffn* const* layers, ts_predictor* const* preds,
                                           int n_layers, float* h, int batch, const int* K,
                                           int32_t* const* lists) {
    return capture(out, [&](cudaStream_t s) {
        return ts_stack_forward_predicted(layers, preds, n_layers, h, batch, K, lists, s);
    });
}

ts_status ts_graph_capture_stack_fused(ts_graph** out, ts_ffn* const* layers, int n_layers, float* hres,
                                       int batch, const int32_t* const* active_idx, const int* n_active) {
    if (!out) return TS_ERR_INVALID_ARG;
    *out = nullptr;
    if (!layers || n_layers < 1 || !hres || batch < 1) return TS_ERR_INVALID_ARG;
    if (((uintptr_t)hres & 15u) != 0) return TS_ERR_INVALID_ARG;
    const ts_ffn* h0 = layers[0];
    if (!h0) return TS_ERR_INVALID_ARG;
    DeviceInfo dev;
    ts_status st = device_info(&dev);
    if (st != TS_OK) return st;
    const int w = pow2_tokens(batch);
    if (batch > kAccMaxTokens || h0->dt != TS_BF16) return TS_ERR_UNSUPPORTED;
    const int grid = h0->grid[w];
    for (int l = 0; l < n_layers; ++l) {
        const ts_ffn* h = layers[l];
        if (!h || h->d != h0->d || h->dt != h0->dt || batch > h->max_batch) return TS_ERR_INVALID_ARG;
        if (h->grid[w] != grid || use_wide(h, batch)) return TS_ERR_UNSUPPORTED;
        const int32_t* rows = active_idx ? active_idx[l] : nullptr;
        if (rows && !n_active) return TS_ERR_INVALID_ARG;
        st = check_list(h, rows, rows ? n_active[l] : 0);
        if (st != TS_OK) return st;
    }
    if (!stack_fused_supported(h0->d, w, grid, dev.optin_smem)) return TS_ERR_UNSUPPORTED;

    std::vector<FfnLaunch> table(n_layers);
    for (int l = 0; l < n_layers; ++l) {
        const int32_t* rows = active_idx ? active_idx[l] : nullptr;
        FfnLaunch a = ffn_launch(layers[l], batch, rows, rows ? n_active[l] : 0);
        a.h = hres;
        a.norm_from_h = 1;
        a.residual_out = 1;
        a.tok0 = 0;
        a.nt = batch;
        a.bits_tok_base = 0;
        a.partial_ctas = grid;
        table[l] = a;
    }
    const size_t table_bytes = align_up(sizeof(FfnLaunch) * (size_t)n_layers);
    void* mem = nullptr;
    const size_t bar_bytes = align_up(sizeof(unsigned) * (size_t)stack_bar_words(grid));
    if (cudaMalloc(&mem, table_bytes + bar_bytes) != cudaSuccess) {
        cudaGetLastError();
        return TS_ERR_OOM;
    }
    if (cudaMemcpy(mem, table.data(), sizeof(FfnLaunch) * (size_t)n_layers, cudaMemcpyHostToDevice) !=
        cudaSuccess) {
        cudaFree(mem);
        return TS_ERR_CUDA;
    }
    StackLaunch S;
    S.layers = static_cast<const FfnLaunch*>(mem);
    S.n_layers = n_layers;
    S.h = hres;
    S.bar = reinterpret_cast<unsigned*>(static_cast<char*>(mem) + table_bytes);
    S.status = h0->s.status;
    ts_graph* g = nullptr;
    st = capture(&g, [&](cudaStream_t s) {
        // the barrier words and the abort flag start at zero on every replay
        ts_status r = cuda_status(cudaMemsetAsync(S.bar, 0, bar_bytes, s));
        if (r == TS_OK) r = cuda_status(launch_stack_fused(S, h0->d, w, grid, s));
        return r;
    });
    if (st != TS_OK) {
        cudaFree(mem);
        return st;
    }
    g->mem = mem;
    for (int l = 0; l < n_layers; ++l) {
        const int32_t* rows = active_idx ? active_idx[l] : nullptr;
        remember(layers[l], batch, rows, rows ? n_active[l] : 0);
    }
    *out = g;
    return TS_OK;
}

ts_status ts_graph_launch(ts_graph* g, cudaStream_t stream) {
    if (!g || !g->exec) return TS_ERR_INVALID_ARG;
    return cuda_status(cudaGraphLaunch(g->exec, stream));
}

void ts_graph_destroy(ts_graph* g) {
    if (!g) return;
    if (g->exec) cudaGraphExecDestroy(g->exec);
    if (g->graph) cudaGraphDestroy(g->graph);
    if (g->mem) cudaFree(g->mem);
    delete g;
}

}  // extern "C"
