// ts_noalloc.cu -- ts_ffn_forward_noalloc: one dReLU FFN forward (Eq. 1 with
// the dReLU of Eq. 2) that needs no handle and allocates no device memory.
//
// Who needs it: a caller that cannot allocate at the moment it runs the FFN,
// e.g. one running inside a memory pool that is full or must not grow, one
// that must not pay the implicit device synchronisation cudaFree (and at
// times cudaMalloc) performs, or a plain C caller with nowhere to keep a
// handle between calls. The handle API allocates its scratch in
// ts_ffn_create; here the scratch of the two kernels instead lives in one
// fixed-size array of the library's own static device memory, which exists
// as soon as the module is loaded on a device. Its address is looked up once
// per device context with cudaGetSymbolAddress (again if the context is
// recreated) and then handed to the same gate+up and down kernels the handle
// API launches.
//
// What the scratch holds and what must start at zero: c values
// (kMaxPass x m fp32), per-token gate/both bitmaps (batch x nbytes each),
// union bitmaps (nbytes each) and the device status word. Every c value and
// bitmap byte the down kernel reads is written by the gate+up kernel of the
// same call, so only the status word must start at zero; static device
// storage is zero when the module loads, and the kernels only OR flags into
// it. This entry point does not read it back (device-detected list errors
// are not reported here; the entries are skipped as in ts_ffn_forward).
//
// Concurrency: every call on a device uses the same scratch, so calls whose
// executions overlap (different streams, different host threads without
// ordering) race on it. The caller serialises them.
#include <cuda.h>
#include <stdint.h>
#include <string.h>

#include <algorithm>
#include <mutex>

#include "ts_ffn.h"
#include "ts_kernels.cuh"

using namespace tsffn;

namespace {

constexpr int kNoAllocMaxM = 16384;            // neurons per layer (TS_NOALLOC_MAX_M)
constexpr int kNoAllocMaxBatch = kMaxBatch;    // tokens per call (TS_NOALLOC_MAX_BATCH)
constexpr size_t kSlab = 256;
constexpr size_t slab(size_t n) { return (n + kSlab - 1) / kSlab * kSlab; }
constexpr size_t kNbytesMax = (size_t)(kNoAllocMaxM + 31) / 32 * 4;
constexpr size_t kOffCval = 0;
constexpr size_t kOffG = kOffCval + slab((size_t)kMaxPass * kNoAllocMaxM * sizeof(float));
constexpr size_t kOffB = kOffG + slab((size_t)kNoAllocMaxBatch * kNbytesMax);
constexpr size_t kOffU = kOffB + slab((size_t)kNoAllocMaxBatch * kNbytesMax);
constexpr size_t kOffUG = kOffU + slab(kNbytesMax);
constexpr size_t kOffStatus = kOffUG + slab(kNbytesMax);
constexpr size_t kScratchBytes = kOffStatus + kSlab;  // ~0.77 MB

static_assert(kNoAllocMaxM == 16384 && kNoAllocMaxBatch == 64,
              "keep TS_NOALLOC_MAX_M / TS_NOALLOC_MAX_BATCH in ts_ffn.h in step");

constexpr int kMaxDevices = 64;

struct NoAllocDevice {
    bool ready = false;
    unsigned long long ctx_id = 0;  // the context the set-up below belongs to
    char* scratch = nullptr;
    int num_sms = 1;
    int optin_smem = 48 * 1024;
};

// The driver's context queries, reached through the runtime so that the
// library does not link libcuda itself.
typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

// Unique id of the current context (0 if none is current or the query fails).
// A context that was destroyed and created again (cudaDeviceReset, or a
// primary context released and retained anew) gets a new id, and the set-up
// of the old one -- the scratch address, the kernels' shared-memory
// attributes -- no longer holds.
unsigned long long current_ctx_id() {
    static CtxGetCurrentFn get_current = nullptr;
    static CtxGetIdFn get_id = nullptr;
    static bool looked_up = false;
    if (!looked_up) {
        void* f0 = nullptr;
        void* f1 = nullptr;
        cudaDriverEntryPointQueryResult q0 = cudaDriverEntryPointSymbolNotFound, q1 = q0;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f0, 12000, cudaEnableDefault, &q0) ==
                cudaSuccess &&
            q0 == cudaDriverEntryPointSuccess)
            get_current = reinterpret_cast<CtxGetCurrentFn>(f0);
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f1, 12000, cudaEnableDefault, &q1) == cudaSuccess &&
            q1 == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<CtxGetIdFn>(f1);
        cudaGetLastError();
        looked_up = true;
    }
    if (get_current == nullptr || get_id == nullptr) return 0;
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return 0;
    if (get_id(ctx, &id) != CUDA_SUCCESS) return 0;
    return id;
}

std::mutex g_setup_mu;
NoAllocDevice g_dev[kMaxDevices];

}  // namespace

// The scratch: static device memory of the library, never allocated or freed.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

namespace {

// First call on a device (with that device current), and the first call
// after that device's context was recreated: find the scratch, read the
// device facts and set the kernels' shared-memory attributes.
ts_status setup_device(NoAllocDevice** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return TS_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return TS_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_setup_mu);
    NoAllocDevice& nd = g_dev[dev];
    const unsigned long long id = current_ctx_id();
    if (!nd.ready || id == 0 || id != nd.ctx_id) {
        nd.ready = false;
        void* p = nullptr;
        // also creates the device's primary context if none is current yet
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) {
            cudaGetLastError();
            return TS_ERR_CUDA;
        }
        nd.ctx_id = current_ctx_id();
        if (cudaDeviceGetAttribute(&nd.num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&nd.optin_smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
                cudaSuccess)
            return TS_ERR_CUDA;
        if (prepare_gate_up(nd.optin_smem) != cudaSuccess || prepare_down() != cudaSuccess)
            return TS_ERR_CUDA;
        nd.scratch = static_cast<char*>(p);
        nd.ready = true;
    }
    *out = &nd;
    return TS_OK;
}

}  // namespace

extern "C" ts_status ts_ffn_forward_noalloc(int d, int m, ts_dtype wdtype, const void* w_gate,
                                            const void* w_up, const void* w_down, const void* x,
                                            int batch, float* y, cudaStream_t stream,
                                            const int32_t* active_idx, int n_active) {
    if (d < 1 || m < 1 || batch < 0) return TS_ERR_INVALID_ARG;
    if (wdtype != TS_F32 && wdtype != TS_BF16) return TS_ERR_INVALID_ARG;
    if (!w_gate || !w_up || !w_down) return TS_ERR_INVALID_ARG;
    const int elem = wdtype == TS_BF16 ? 2 : 4;
    if ((((uintptr_t)w_gate | (uintptr_t)w_up | (uintptr_t)w_down) & 15u) != 0) return TS_ERR_INVALID_ARG;
    if (((size_t)d * elem) % 16 != 0) return TS_ERR_INVALID_ARG;
    if (active_idx != nullptr && (n_active < 0 || n_active > m)) return TS_ERR_INVALID_ARG;
    if (m > kNoAllocMaxM || batch > kNoAllocMaxBatch) return TS_ERR_UNSUPPORTED;
    if (batch == 0) return TS_OK;
    if (!x || !y) return TS_ERR_INVALID_ARG;

    NoAllocDevice* nd = nullptr;
    ts_status st = setup_device(&nd);
    if (st != TS_OK) return st;
    {
        int slots, slot_bytes, xs_stride;
        size_t smem;
        if (gate_up_config(wdtype, d, std::min(batch, kMaxPass), nd->optin_smem, &slots, &slot_bytes,
                           &xs_stride, &smem) != 0)
            return TS_ERR_UNSUPPORTED;
    }

    FfnLaunch a;
    memset(&a, 0, sizeof a);
    a.d = d;
    a.m = m;
    a.elem_bytes = elem;
    a.row_bytes = d * elem;
    a.rows = active_idx;
    a.n_rows = active_idx ? n_active : m;
    a.batch = batch;
    a.x = x;
    a.y = y;
    a.n_experts = 1;
    a.ex[0] = ExpertPtrs{w_gate, w_up, w_down};
    a.top_k = 1;
    a.cval = reinterpret_cast<float*>(nd->scratch + kOffCval);
    a.cval_tok_stride = m;
    a.nbytes = (m + 31) / 32 * 4;
    a.gbits = reinterpret_cast<uint8_t*>(nd->scratch + kOffG);
    a.bbits = reinterpret_cast<uint8_t*>(nd->scratch + kOffB);
    a.ubits = reinterpret_cast<uint8_t*>(nd->scratch + kOffU);
    a.ugbits = reinterpret_cast<uint8_t*>(nd->scratch + kOffUG);
    a.status = reinterpret_cast<unsigned*>(nd->scratch + kOffStatus);
    const int grid = std::max(1, std::min(nd->num_sms, (m + kChunk - 1) / kChunk));

    for (int t0 = 0; t0 < batch; t0 += kMaxPass) {
        const int nt = std::min(kMaxPass, batch - t0);
        // widths of at least 4 gather W_down in the down kernel and need no
        // per-CTA partial buffer
        const int w = nt <= 4 ? 4 : 8;
        a.tok0 = t0;
        a.nt = nt;
        a.bits_tok_base = t0;
        if (launch_gate_up(a, wdtype, w, grid, stream, true) != cudaSuccess) return TS_ERR_CUDA;
        if (launch_down(a, wdtype, w, stream, true) != cudaSuccess) return TS_ERR_CUDA;
    }
    return TS_OK;
}
