// statekv_frame_attention_noalloc: the frame attention with importance for
// one (stream, layer), for callers that cannot allocate device memory.
//
// Callers such as plugins running inside a host application's fixed memory
// budget, or code paths that must not call cudaMalloc (it can synchronise the
// device and is not allowed while another component is capturing a stream),
// still need the attention kernel's scratch: the per-query-tile importance
// partials, the per-head state counts and a status word.  Here that scratch is
// a set of file-scope __device__ arrays of fixed size, resident on every GPU
// that loads the library until the process exits.  The caller passes only its
// inputs and outputs.
//
// Host code must not hand the arrays' names to a kernel: on the host they are
// stand-ins, not device addresses.  The first call on each device looks their
// device addresses up with cudaGetSymbolAddress (with that device current)
// and caches them; that first call should happen before any stream capture.
//
// Every call shares the same scratch, which keeps the previous call's
// contents: the counts and the status word are rewritten at the start of
// each call, and the kernels write every partial they later read.  Calls that
// overlap on the GPU (different streams or threads, no ordering) race on the
// scratch.  Each call synchronises its stream before returning, so the stream
// must not be under capture (refused), and a caller that runs while another
// component captures should pass a cudaStreamNonBlocking stream: a blocking
// stream, the legacy default stream among them, synchronises implicitly with
// the capturing stream, which invalidates that capture.
#include "../../include/statekv.h"
#include "statekv_kernels.cuh"

#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <mutex>

namespace statekv {
namespace {

// Scratch limits: partials for Hkv * MT * (B + T) floats and counts for up to
// kNoAllocMaxKV KV heads (MT = ceil(G * T / 128) query tiles per KV head).
constexpr size_t kNoAllocMaxPartials = 1u << 20;  // 4 MB of fp32 partials
constexpr int kNoAllocMaxKV = 64;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) float g_partials[kNoAllocMaxPartials];
static __device__ __align__(256) int32_t g_counts[kNoAllocMaxKV];
static __device__ __align__(256) int32_t g_status[1];

struct ScratchAddrs {
    float* partials = nullptr;
    int32_t* counts = nullptr;
    int32_t* status = nullptr;
    bool ready = false;
};

std::mutex g_setup_mu;
ScratchAddrs g_addrs[kMaxDevices];

// Device addresses of the scratch arrays on the current device (set-up on
// the first call per device).
cudaError_t scratch_for_current_device(ScratchAddrs* out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_setup_mu);
    ScratchAddrs& a = g_addrs[dev];
    if (!a.ready) {
        void* p = nullptr;
        if ((e = cudaGetSymbolAddress(&p, g_partials)) != cudaSuccess) return e;
        a.partials = static_cast<float*>(p);
        if ((e = cudaGetSymbolAddress(&p, g_counts)) != cudaSuccess) return e;
        a.counts = static_cast<int32_t*>(p);
        if ((e = cudaGetSymbolAddress(&p, g_status)) != cudaSuccess) return e;
        a.status = static_cast<int32_t*>(p);
        if ((e = attn_prepare(64)) != cudaSuccess) return e;
        if ((e = attn_prepare(128)) != cudaSuccess) return e;
        a.ready = true;
    }
    *out = a;
    return cudaSuccess;
}

__global__ void noalloc_reset(int32_t* counts, int hkv, int32_t count, int32_t* status)
{
    const int i = threadIdx.x;
    if (i < hkv) counts[i] = count;
    if (i == 0) status[0] = 0;
}

// importance[h][c] = sum over query tiles of the partials (fixed order);
// state columns past the valid count are 0.
__global__ void noalloc_importance(const float* __restrict__ partials, float* __restrict__ imp,
                                   int Hkv, int MT, int P, int B, int count)
{
    const int n = Hkv * P;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        const int h = i / P, c = i - h * P;
        float s = 0.f;
        if (c >= B || c < count)
            for (int mt = 0; mt < MT; ++mt) s += partials[(static_cast<size_t>(h) * MT + mt) * P + c];
        imp[i] = s;
    }
}

// The frame's K or V ([T][Hkv][D]: boxes of one head x 128 tokens) or the
// state's ([Hkv][B][D]: boxes of 128 slots of one head), as the handle path
// maps them for one (stream, layer).
bool noalloc_map(CUtensorMap* m, const void* base, cuuint64_t d0, cuuint64_t d1, cuuint64_t d2,
                 cuuint32_t b1, cuuint32_t b2)
{
    const cuuint64_t dims[4] = {d0, d1, d2, 1};
    const cuuint64_t strides[3] = {d0 * 2, d0 * d1 * 2, d0 * d1 * d2 * 2};
    const cuuint32_t box[4] = {64, b1, b2, 1};
    return encode_4d(m, base, dims, strides, box);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace statekv

using namespace statekv;

extern "C" statekv_status statekv_frame_attention_noalloc(
    const statekv_config* cfg, const void* q, const void* k, const void* v, const void* state_k,
    const void* state_v, int32_t state_count, void* out, float* importance, statekv_stream stream)
{
    if (!cfg || !q || !k || !v || !out || !importance) return STATEKV_ERR_INVALID_ARG;
    const int Hq = cfg->num_q_heads, Hkv = cfg->num_kv_heads, D = cfg->head_dim;
    const int T = cfg->tokens_per_frame, B = cfg->state_capacity;
    if (Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || T < 1 || B < 0 || state_count < 0 ||
        state_count > B || (cfg->causal_in_frame != 0 && cfg->causal_in_frame != 1) ||
        !(cfg->softmax_scale >= 0.f) || !std::isfinite(cfg->softmax_scale))
        return STATEKV_ERR_INVALID_ARG;
    if (B > 0 && (!state_k || !state_v || !aligned16(state_k) || !aligned16(state_v)))
        return STATEKV_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out) ||
        (reinterpret_cast<uintptr_t>(importance) & 3u))
        return STATEKV_ERR_INVALID_ARG;
    if (D != 64 && D != 128) return STATEKV_ERR_UNSUPPORTED;
    const int G = Hq / Hkv;
    // sizes beyond what the kernels or the fixed scratch take are refused
    // before anything is computed from them in int
    if (T > kMaxFrameTokens || Hkv > kNoAllocMaxKV ||
        static_cast<long long>(G) * T > 0x7FFFFFFFll)
        return STATEKV_ERR_UNSUPPORTED;
    const long long MT = (static_cast<long long>(G) * T + kBM - 1) / kBM;
    const long long P = static_cast<long long>(B) + T;
    if (static_cast<long long>(Hkv) * MT * P > static_cast<long long>(kNoAllocMaxPartials))
        return STATEKV_ERR_UNSUPPORTED;

    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    // The call waits for its own work (below), which a stream being captured
    // cannot do; refuse such a stream before enqueueing anything.
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st, &cap) != cudaSuccess || cap != cudaStreamCaptureStatusNone) {
        cudaGetLastError();  // a refused query leaves no sticky error behind
        return STATEKV_ERR_INVALID_ARG;
    }
    ScratchAddrs s;
    if (scratch_for_current_device(&s) != cudaSuccess) return STATEKV_ERR_CUDA;

    CUtensorMap tm_sk{}, tm_sv{}, tm_fk{}, tm_fv{};
    if (!noalloc_map(&tm_fk, k, D, Hkv, T, 1, kBN) || !noalloc_map(&tm_fv, v, D, Hkv, T, 1, kBN))
        return STATEKV_ERR_CUDA;
    if (B > 0 && (!noalloc_map(&tm_sk, state_k, D, B, Hkv, kBN, 1) ||
                  !noalloc_map(&tm_sv, state_v, D, B, Hkv, kBN, 1)))
        return STATEKV_ERR_CUDA;

    noalloc_reset<<<1, kNoAllocMaxKV, 0, st>>>(s.counts, Hkv, state_count, s.status);
    if (cudaGetLastError() != cudaSuccess) return STATEKV_ERR_CUDA;

    AttnParams p{};
    p.q = static_cast<const __nv_bfloat16*>(q);
    p.out = static_cast<__nv_bfloat16*>(out);
    p.partials = s.partials;
    p.counts = s.counts;
    p.status = s.status;
    p.units = UnitRange{0, 0, 1, 1};
    p.T = T;
    p.Hq = Hq;
    p.Hkv = Hkv;
    p.G = G;
    p.B = B;
    p.P = static_cast<int>(P);
    p.MT = static_cast<int>(MT);
    p.causal = cfg->causal_in_frame;
    p.count_mul = 1;
    const float scale =
        cfg->softmax_scale > 0.f ? cfg->softmax_scale : 1.0f / std::sqrt(static_cast<float>(D));
    p.scale_log2 = scale * 1.4426950408889634f;
    p.watchdog_ns = 1000000ull * (cfg->watchdog_ms ? cfg->watchdog_ms : 2000u);
    if (launch_attn(D, tm_sk, tm_sv, tm_fk, tm_fv, p, 1, st) != cudaSuccess) return STATEKV_ERR_CUDA;
    noalloc_importance<<<(Hkv * static_cast<int>(P) + 255) / 256, 256, 0, st>>>(
        s.partials, importance, Hkv, static_cast<int>(MT), static_cast<int>(P), B, state_count);
    if (cudaGetLastError() != cudaSuccess) return STATEKV_ERR_CUDA;
    // The call completes before it returns, so it can report its own device
    // status (an expired wait leaves out / importance unspecified).
    int32_t word = 0;
    if (cudaMemcpyAsync(&word, s.status, sizeof(word), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess)
        return STATEKV_ERR_CUDA;
    if (word != 0)
        return (word & 0xFF) == DEV_TIMEOUT_ATTN ? STATEKV_ERR_DEVICE_TIMEOUT
                                                 : STATEKV_ERR_DEVICE_FAULT;
    return STATEKV_OK;
}
