// Host runtime behind include/statekv.h: configuration checks, arena
// carve-up, TMA descriptor encoding, launch sequencing and profiling.
//
// Per call, in stream order:  K4 append -> K1 attention -> K3 select/gather.
// K4 reads the per-head frame counter before K3 advances it; K1 reads the
// state before K3 rewrites it.
#include "../../include/statekv.h"
#include "statekv_kernels.cuh"

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

using namespace statekv;

namespace {

constexpr size_t kAlign = 256;
constexpr int kProfPairs = 3 * 4096;

size_t round_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// Debug builds put a guard band of kGuardBytes after every arena region,
// filled with kGuardFill at init and compared by statekv_debug_check.
constexpr size_t kGuard = STATEKV_DEBUG_CHECKS ? kGuardBytes : 0;

struct Layout {
    size_t state_k, state_v, positions, counts, frames, text, cache_k, cache_v, partials;
    struct Staging {
        size_t q, k, v, out, imp;
    } stg[2];  // host-buffer calls: two frames, so copies overlap the steps
    GuardList guards;
    size_t total;
};

struct Derived {
    int G, MT, P, SL;
    long long cap;
    float scale;
};

statekv_status check_config(const statekv_config* c, Derived* d)
{
    if (!c) return STATEKV_ERR_INVALID_ARG;
    if (c->num_streams < 1 || c->num_layers < 1 || c->num_q_heads < 1 || c->num_kv_heads < 1 ||
        c->num_q_heads % c->num_kv_heads != 0 || c->head_dim < 1 || c->tokens_per_frame < 1 ||
        c->state_capacity < 0 || c->max_frames < 1 ||
        (c->causal_in_frame != 0 && c->causal_in_frame != 1) ||
        (c->host_staging != 0 && c->host_staging != 1) ||
        (c->selection < 0 || c->selection > 2) || !(c->softmax_scale >= 0.f) ||
        !std::isfinite(c->softmax_scale))
        return STATEKV_ERR_INVALID_ARG;
    if (static_cast<long long>(c->max_frames) * c->tokens_per_frame > 0x7FFFFFFFll)
        return STATEKV_ERR_INVALID_ARG;  // positions are int32
    if (c->head_dim != 64 && c->head_dim != 128) return STATEKV_ERR_UNSUPPORTED;
    if (c->tokens_per_frame > kMaxFrameTokens) return STATEKV_ERR_UNSUPPORTED;
    if (static_cast<long long>(c->state_capacity) + c->tokens_per_frame > kMaxPool)
        return STATEKV_ERR_UNSUPPORTED;
    if (c->num_kv_heads > 65535 || static_cast<long long>(c->num_streams) * c->num_layers > 65535)
        return STATEKV_ERR_UNSUPPORTED;
    d->G = c->num_q_heads / c->num_kv_heads;
    d->MT = static_cast<int>((static_cast<long long>(d->G) * c->tokens_per_frame + kBM - 1) / kBM);
    d->P = c->state_capacity + c->tokens_per_frame;
    d->SL = c->num_streams * c->num_layers;
    d->cap = static_cast<long long>(c->max_frames) * c->tokens_per_frame;
    d->scale = c->softmax_scale > 0.f ? c->softmax_scale
                                      : 1.0f / std::sqrt(static_cast<float>(c->head_dim));
    return STATEKV_OK;
}

Layout make_layout(const statekv_config& c, const Derived& d)
{
    Layout L{};
    const size_t heads = static_cast<size_t>(d.SL) * c.num_kv_heads;
    const size_t D = c.head_dim, B = c.state_capacity, T = c.tokens_per_frame;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        const size_t at = off;
        off += round_up(bytes);
        if (kGuard > 0 && L.guards.n < kMaxGuards) {
            L.guards.off[L.guards.n++] = off;
            off += kGuard;
        }
        return at;
    };
    L.state_k = take(heads * B * D * 2);
    L.state_v = take(heads * B * D * 2);
    L.positions = take(heads * B * 4);
    L.counts = take(heads * 4);
    L.frames = take(heads * 4);
    L.text = take(heads * 4);  // decode-cache rows appended after the video frames
    L.cache_k = take(heads * static_cast<size_t>(d.cap) * D * 2);
    L.cache_v = take(heads * static_cast<size_t>(d.cap) * D * 2);
    // importance partials of a frame step; a decode step's split-K partials
    // use the same bytes (the two never overlap in time on a handle)
    L.partials = take(std::max(heads * d.MT * static_cast<size_t>(d.P) * 4,
                               heads * kDecodeMaxChunks * kDecodeRows * (static_cast<size_t>(D) + 2) * 4));
    if (c.host_staging) {
        for (auto& g : L.stg) {
            g.q = take(static_cast<size_t>(d.SL) * T * c.num_q_heads * D * 2);
            g.k = take(heads * T * D * 2);
            g.v = take(heads * T * D * 2);
            g.out = take(static_cast<size_t>(d.SL) * T * c.num_q_heads * D * 2);
            g.imp = take(heads * static_cast<size_t>(d.P) * 4);
        }
    }
    L.total = off;
    return L;
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

struct ProfRec {
    cudaEvent_t a, b;
    int kind;
};

}  // namespace

namespace statekv {

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

bool tma_encode_available() { return encode_fn() != nullptr; }

bool encode_4d(CUtensorMap* m, const void* base, const cuuint64_t dims[4],
               const cuuint64_t strides_bytes[3], const cuuint32_t box[4])
{
    auto fn = encode_fn();
    if (!fn) return false;
    const cuuint32_t es[4] = {1, 1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides_bytes,
              box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace statekv

struct statekv_handle {
    statekv_config cfg;
    Derived d;
    Layout lay;
    uint8_t* arena;
    std::vector<int32_t> frames_host;  // [S*L]
    std::vector<int32_t> text_host;    // [S*L]: tokens appended by statekv_decode_step
    CUtensorMap tm_sk, tm_sv;  // state rows, [S*L][Hkv][B][D]
    CUtensorMap tm_ck, tm_cv;  // decode-cache rows, [S*L][Hkv][cap][D], boxes of 128 keys
    CUtensorMap tm_dk, tm_dv;  // the same with boxes of kDecodeKeyBox keys (decode kernel)
    volatile int32_t* status_host;
    int32_t* status_dev;
    bool prof_on;
    size_t prof_used;
    std::vector<ProfRec> prof;
    // The decode-cache append runs on a side stream forked from the call's
    // stream and joined before the selection: it depends on nothing the
    // attention kernel writes, so it fills SMs the attention grid leaves idle.
    cudaStream_t side = nullptr;
    cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
    // Pipelined host-buffer frames: copies in and out run on their own
    // streams; per staging set, "copied in", "step done", "copied out".
    cudaStream_t cin = nullptr, cout = nullptr;
    cudaEvent_t ev_start = nullptr, ev_in[2] = {}, ev_comp[2] = {}, ev_out[2] = {};

    template <class T>
    T* at(size_t off) const { return reinterpret_cast<T*>(arena + off); }
};

namespace {

bool create_streams(statekv_handle* h)
{
    bool ok = cudaStreamCreateWithFlags(&h->side, cudaStreamNonBlocking) == cudaSuccess &&
              cudaStreamCreateWithFlags(&h->cin, cudaStreamNonBlocking) == cudaSuccess &&
              cudaStreamCreateWithFlags(&h->cout, cudaStreamNonBlocking) == cudaSuccess;
    for (cudaEvent_t* e : {&h->ev_fork, &h->ev_join, &h->ev_start, &h->ev_in[0], &h->ev_in[1],
                           &h->ev_comp[0], &h->ev_comp[1], &h->ev_out[0], &h->ev_out[1]})
        ok = ok && cudaEventCreateWithFlags(e, cudaEventDisableTiming) == cudaSuccess;
    return ok;
}

void release_streams(statekv_handle* h)
{
    for (cudaEvent_t e : {h->ev_fork, h->ev_join, h->ev_start, h->ev_in[0], h->ev_in[1],
                          h->ev_comp[0], h->ev_comp[1], h->ev_out[0], h->ev_out[1]})
        if (e) cudaEventDestroy(e);
    for (cudaStream_t st : {h->side, h->cin, h->cout})
        if (st) cudaStreamDestroy(st);
}

statekv_status device_status(int32_t word)
{
    if (word == 0) return STATEKV_OK;
    const int kind = word & 0xFF;
    return kind == DEV_TIMEOUT_ATTN || kind == DEV_TIMEOUT_GEMM || kind == DEV_TIMEOUT_DECODE
               ? STATEKV_ERR_DEVICE_TIMEOUT
               : STATEKV_ERR_DEVICE_FAULT;
}

statekv_status check_args(const statekv_handle* h, const statekv_frame_args* a, bool host)
{
    if (!h || !a) return STATEKV_ERR_INVALID_ARG;
    const statekv_config& c = h->cfg;
    if (a->stream_count < 1 || a->layer_count < 1 || a->stream_begin < 0 || a->layer_begin < 0 ||
        a->stream_begin + a->stream_count > c.num_streams ||
        a->layer_begin + a->layer_count > c.num_layers)
        return STATEKV_ERR_INVALID_ARG;
    if (!a->q || !a->k || !a->v || !a->out) return STATEKV_ERR_INVALID_ARG;
    if (!host) {
        if (!aligned(a->q, 16) || !aligned(a->k, 16) || !aligned(a->v, 16) || !aligned(a->out, 16) ||
            (a->importance && !aligned(a->importance, 4)))
            return STATEKV_ERR_INVALID_ARG;
    }
    if (host && !c.host_staging) return STATEKV_ERR_INVALID_ARG;
    if (c.selection == 1 && a->importance) return STATEKV_ERR_INVALID_ARG;  // none computed
    if (*h->status_host != 0) return device_status(*h->status_host);
    for (int s = a->stream_begin; s < a->stream_begin + a->stream_count; ++s)
        for (int l = a->layer_begin; l < a->layer_begin + a->layer_count; ++l) {
            const size_t unit = static_cast<size_t>(s) * c.num_layers + l;
            if (h->text_host[unit] > 0) return STATEKV_ERR_INVALID_ARG;  // video closed
            if (h->frames_host[unit] >= c.max_frames) return STATEKV_ERR_CACHE_FULL;
        }
    return STATEKV_OK;
}

template <class F>
cudaError_t timed(statekv_handle* h, int kind, cudaStream_t st, F&& launch)
{
    ProfRec* r = nullptr;
    if (h->prof_on && h->prof_used < h->prof.size()) {
        r = &h->prof[h->prof_used++];
        r->kind = kind;
        cudaEventRecord(r->a, st);
    }
    cudaError_t e = launch();
    if (r) cudaEventRecord(r->b, st);
    return e;
}

statekv_status run_step(statekv_handle* h, const statekv_frame_args& a, cudaStream_t st)
{
    const statekv_config& c = h->cfg;
    const Derived& d = h->d;
    const int U = a.stream_count * a.layer_count;
    const int D = c.head_dim, T = c.tokens_per_frame, Hkv = c.num_kv_heads;
    const UnitRange ur{a.stream_begin, a.layer_begin, a.layer_count, c.num_layers};

    CUtensorMap tm_fk, tm_fv;
    {
        const cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(Hkv),
                                    static_cast<cuuint64_t>(T), static_cast<cuuint64_t>(U)};
        const cuuint64_t strides[3] = {static_cast<cuuint64_t>(D) * 2,
                                       static_cast<cuuint64_t>(Hkv) * D * 2,
                                       static_cast<cuuint64_t>(T) * Hkv * D * 2};
        const cuuint32_t box[4] = {64, 1, static_cast<cuuint32_t>(kBN), 1};
        if (!encode_4d(&tm_fk, a.k, dims, strides, box) ||
            !encode_4d(&tm_fv, a.v, dims, strides, box))
            return STATEKV_ERR_CUDA;
    }
    int32_t* counts = h->at<int32_t>(h->lay.counts);
    int32_t* frames = h->at<int32_t>(h->lay.frames);
    float* partials = h->at<float>(h->lay.partials);

    AppendParams ap{};
    ap.k = static_cast<const __nv_bfloat16*>(a.k);
    ap.v = static_cast<const __nv_bfloat16*>(a.v);
    ap.cache_k = h->at<__nv_bfloat16>(h->lay.cache_k);
    ap.cache_v = h->at<__nv_bfloat16>(h->lay.cache_v);
    ap.frames = frames;
    ap.units = ur;
    ap.U = U;
    ap.T = T;
    ap.Hkv = Hkv;
    ap.D = D;
    ap.row_mul = T;
    ap.cap = d.cap;
    ap.status = h->status_dev;
    // append on the side stream; it reads the frame counters, so the join
    // comes before the selection kernel advances them
    if (cudaEventRecord(h->ev_fork, st) != cudaSuccess ||
        cudaStreamWaitEvent(h->side, h->ev_fork, 0) != cudaSuccess ||
        timed(h, 0, h->side, [&] { return launch_append(ap, h->side); }) != cudaSuccess ||
        cudaEventRecord(h->ev_join, h->side) != cudaSuccess)
        return STATEKV_ERR_CUDA;

    AttnParams pa{};
    pa.q = static_cast<const __nv_bfloat16*>(a.q);
    pa.out = static_cast<__nv_bfloat16*>(a.out);
    pa.partials = c.selection != 1 ? partials : nullptr;  // recency: no importance
    pa.counts = counts;
    pa.status = h->status_dev;
    pa.units = ur;
    pa.T = T;
    pa.Hq = c.num_q_heads;
    pa.Hkv = Hkv;
    pa.G = d.G;
    pa.B = c.state_capacity;
    pa.P = d.P;
    pa.MT = d.MT;
    pa.causal = c.causal_in_frame;
    pa.count_mul = 1;
    pa.scale_log2 = d.scale * 1.4426950408889634f;
    pa.watchdog_ns = 1000000ull * (c.watchdog_ms ? c.watchdog_ms : 2000u);
    const cudaError_t ek =
        timed(h, 1, st, [&] { return launch_attn(D, h->tm_sk, h->tm_sv, tm_fk, tm_fv, pa, U, st); });
    const cudaError_t ej = cudaStreamWaitEvent(st, h->ev_join, 0);  // the append is done
    if (ek != cudaSuccess || ej != cudaSuccess) return STATEKV_ERR_CUDA;

    if (c.selection == 1) {
        RecencyParams pr{};
        pr.k = ap.k;
        pr.v = ap.v;
        pr.state_k = h->at<__nv_bfloat16>(h->lay.state_k);
        pr.state_v = h->at<__nv_bfloat16>(h->lay.state_v);
        pr.positions = h->at<int32_t>(h->lay.positions);
        pr.counts = counts;
        pr.frames = frames;
        pr.units = ur;
        pr.U = U;
        pr.T = T;
        pr.Hkv = Hkv;
        pr.D = D;
        pr.B = c.state_capacity;
        if (timed(h, 2, st, [&] { return launch_recency(pr, st); }) != cudaSuccess)
            return STATEKV_ERR_CUDA;
    } else {
    SelectParams ps{};
    ps.partials = partials;
    ps.importance = a.importance;
    ps.k = ap.k;
    ps.v = ap.v;
    ps.state_k = h->at<__nv_bfloat16>(h->lay.state_k);
    ps.state_v = h->at<__nv_bfloat16>(h->lay.state_v);
    ps.positions = h->at<int32_t>(h->lay.positions);
    ps.counts = counts;
    ps.frames = frames;
    ps.status = h->status_dev;
    ps.units = ur;
    ps.T = T;
    ps.Hkv = Hkv;
    ps.D = D;
    ps.B = c.state_capacity;
    ps.P = d.P;
    ps.MT = d.MT;
    ps.shared = c.selection == 2 ? 1 : 0;
    if (timed(h, 2, st, [&] { return launch_select(ps, U, st); }) != cudaSuccess)
        return STATEKV_ERR_CUDA;
    }

    for (int s = a.stream_begin; s < a.stream_begin + a.stream_count; ++s)
        for (int l = a.layer_begin; l < a.layer_begin + a.layer_count; ++l)
            ++h->frames_host[static_cast<size_t>(s) * c.num_layers + l];
    return STATEKV_OK;
}

// Exact full self-attention of the frame over every token of the decode cache
// (the frames processed so far, all visible) followed by the frame's own
// tokens (causal as configured): the attention kernel with the cache as its
// key prefix, no importance, no change to any state.
statekv_status run_full(statekv_handle* h, const statekv_frame_args& a, cudaStream_t st,
                        float* partials = nullptr, long long Bp = 0)
{
    const statekv_config& c = h->cfg;
    const Derived& d = h->d;
    const int U = a.stream_count * a.layer_count;
    const int D = c.head_dim, T = c.tokens_per_frame, Hkv = c.num_kv_heads;
    CUtensorMap tm_fk, tm_fv;
    {
        const cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(Hkv),
                                    static_cast<cuuint64_t>(T), static_cast<cuuint64_t>(U)};
        const cuuint64_t strides[3] = {static_cast<cuuint64_t>(D) * 2,
                                       static_cast<cuuint64_t>(Hkv) * D * 2,
                                       static_cast<cuuint64_t>(T) * Hkv * D * 2};
        const cuuint32_t box[4] = {64, 1, static_cast<cuuint32_t>(kBN), 1};
        if (!encode_4d(&tm_fk, a.k, dims, strides, box) ||
            !encode_4d(&tm_fv, a.v, dims, strides, box))
            return STATEKV_ERR_CUDA;
    }
    AttnParams pa{};
    pa.q = static_cast<const __nv_bfloat16*>(a.q);
    pa.out = static_cast<__nv_bfloat16*>(a.out);
    pa.partials = partials;  // with partials: key j of the cache at column j, frame token t at Bp + t
    pa.counts = h->at<int32_t>(h->lay.frames);  // keys = frames * T + text rows
    pa.count_add = h->at<int32_t>(h->lay.text);
    pa.status = h->status_dev;
    pa.units = UnitRange{a.stream_begin, a.layer_begin, a.layer_count, c.num_layers};
    pa.T = T;
    pa.Hq = c.num_q_heads;
    pa.Hkv = Hkv;
    pa.G = d.G;
    pa.B = partials ? static_cast<int>(Bp) : 1;  // 1: no importance pool
    pa.P = partials ? static_cast<int>(Bp + T) : 0;
    pa.MT = d.MT;
    pa.causal = c.causal_in_frame;
    pa.count_mul = T;
    pa.scale_log2 = d.scale * 1.4426950408889634f;
    pa.watchdog_ns = 1000000ull * (c.watchdog_ms ? c.watchdog_ms : 2000u);
    if (timed(h, 1, st, [&] { return launch_attn(D, h->tm_ck, h->tm_cv, tm_fk, tm_fv, pa, U, st); }) !=
        cudaSuccess)
        return STATEKV_ERR_CUDA;
    return STATEKV_OK;
}

// Decoding over the detailed cache: n new tokens per (stream, layer) attend to
// every row of the decode cache (video frames, then earlier decoded tokens)
// and causally to each other; their K/V rows are then appended to the cache.
statekv_status run_decode(statekv_handle* h, const statekv_decode_args& a, cudaStream_t st)
{
    const statekv_config& c = h->cfg;
    const Derived& d = h->d;
    const int U = a.stream_count * a.layer_count;
    const int D = c.head_dim, T = c.tokens_per_frame, Hkv = c.num_kv_heads, n = a.num_tokens;
    const UnitRange ur{a.stream_begin, a.layer_begin, a.layer_count, c.num_layers};
    int32_t* frames = h->at<int32_t>(h->lay.frames);
    int32_t* text = h->at<int32_t>(h->lay.text);
    AppendParams ap{};
    ap.k = static_cast<const __nv_bfloat16*>(a.k);
    ap.v = static_cast<const __nv_bfloat16*>(a.v);
    ap.cache_k = h->at<__nv_bfloat16>(h->lay.cache_k);
    ap.cache_v = h->at<__nv_bfloat16>(h->lay.cache_v);
    ap.frames = frames;
    ap.row_add = text;
    ap.units = ur;
    ap.U = U;
    ap.T = n;
    ap.Hkv = Hkv;
    ap.D = D;
    ap.row_mul = T;
    ap.cap = d.cap;
    ap.status = h->status_dev;
    if (n * d.G <= kDecodeRows) {
        // A few rows: the new tokens' K/V go into the cache first, then the
        // one-pass split-K kernel reads every key once from the cache.
        long long maxlen = 0;
        for (int s = a.stream_begin; s < a.stream_begin + a.stream_count; ++s)
            for (int l = a.layer_begin; l < a.layer_begin + a.layer_count; ++l) {
                const size_t unit = static_cast<size_t>(s) * c.num_layers + l;
                maxlen = std::max(maxlen, static_cast<long long>(h->frames_host[unit]) * T +
                                              h->text_host[unit] + n);
            }
        // chunk count: the one whose waves of CTAs (one per SM) take the least
        // time, counting each CTA's fixed cost as ~512 keys of streaming
        DecodeParams dp{};
        {
            const long long units = static_cast<long long>(U) * Hkv, sms = device_sm_count();
            long long best = -1;
            for (int nc = 1; nc <= kDecodeMaxChunks; ++nc) {
                const long long ck = std::max(128ll, ((maxlen + nc - 1) / nc + 127) / 128 * 128);
                const long long used = (maxlen + ck - 1) / ck;
                const long long waves = (units * used + sms - 1) / sms;
                const long long cost = waves * (ck + 512);
                if (best < 0 || cost < best) {
                    best = cost;
                    dp.ck = static_cast<int>(ck);
                    dp.nchunk = static_cast<int>(used);
                }
            }
        }
        dp.q = static_cast<const __nv_bfloat16*>(a.q);
        dp.out = static_cast<__nv_bfloat16*>(a.out);
        dp.cache_k = ap.cache_k;
        dp.cache_v = ap.cache_v;
        dp.frames = frames;
        dp.text = text;
        dp.part_o = h->at<float>(h->lay.partials);
        dp.part_ml = dp.part_o + static_cast<size_t>(U) * Hkv * dp.nchunk * kDecodeRows * D;
        dp.units = ur;
        dp.n = n;
        dp.G = d.G;
        dp.Hq = c.num_q_heads;
        dp.Hkv = Hkv;
        dp.T = T;
        dp.cap = d.cap;
        dp.scale_log2 = d.scale * 1.4426950408889634f;
        dp.status = h->status_dev;
        dp.watchdog_ns = 1000000ull * (c.watchdog_ms ? c.watchdog_ms : 2000u);
        if (timed(h, 0, st, [&] { return launch_append(ap, st); }) != cudaSuccess ||
            timed(h, 1, st, [&] { return launch_decode(h->tm_dk, h->tm_dv, dp, D, U, st); }) != cudaSuccess ||
            launch_advance(text, ur, U, Hkv, n, st) != cudaSuccess)
            return STATEKV_ERR_CUDA;
        for (int s = a.stream_begin; s < a.stream_begin + a.stream_count; ++s)
            for (int l = a.layer_begin; l < a.layer_begin + a.layer_count; ++l)
                h->text_host[static_cast<size_t>(s) * c.num_layers + l] += n;
        return STATEKV_OK;
    }
    CUtensorMap tm_nk, tm_nv;
    {
        const cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(Hkv),
                                    static_cast<cuuint64_t>(n), static_cast<cuuint64_t>(U)};
        const cuuint64_t strides[3] = {static_cast<cuuint64_t>(D) * 2,
                                       static_cast<cuuint64_t>(Hkv) * D * 2,
                                       static_cast<cuuint64_t>(n) * Hkv * D * 2};
        const cuuint32_t box[4] = {64, 1, static_cast<cuuint32_t>(kBN), 1};
        if (!encode_4d(&tm_nk, a.k, dims, strides, box) ||
            !encode_4d(&tm_nv, a.v, dims, strides, box))
            return STATEKV_ERR_CUDA;
    }
    AttnParams pa{};
    pa.q = static_cast<const __nv_bfloat16*>(a.q);
    pa.out = static_cast<__nv_bfloat16*>(a.out);
    pa.partials = nullptr;
    pa.counts = frames;
    pa.count_add = text;
    pa.status = h->status_dev;
    pa.units = ur;
    pa.T = n;
    pa.Hq = c.num_q_heads;
    pa.Hkv = Hkv;
    pa.G = d.G;
    pa.B = 1;  // no importance pool
    pa.P = 0;
    pa.MT = static_cast<int>((static_cast<long long>(d.G) * n + kBM - 1) / kBM);
    pa.causal = 1;
    pa.count_mul = T;
    pa.scale_log2 = d.scale * 1.4426950408889634f;
    pa.watchdog_ns = 1000000ull * (c.watchdog_ms ? c.watchdog_ms : 2000u);
    if (timed(h, 1, st, [&] { return launch_attn(D, h->tm_ck, h->tm_cv, tm_nk, tm_nv, pa, U, st); }) !=
        cudaSuccess)
        return STATEKV_ERR_CUDA;
    if (timed(h, 0, st, [&] { return launch_append(ap, st); }) != cudaSuccess ||
        launch_advance(text, ur, U, Hkv, n, st) != cudaSuccess)
        return STATEKV_ERR_CUDA;
    for (int s = a.stream_begin; s < a.stream_begin + a.stream_count; ++s)
        for (int l = a.layer_begin; l < a.layer_begin + a.layer_count; ++l)
            h->text_host[static_cast<size_t>(s) * c.num_layers + l] += n;
    return STATEKV_OK;
}

}  // namespace

extern "C" {

statekv_status statekv_arena_bytes(const statekv_config* cfg, size_t* bytes)
{
    Derived d;
    const statekv_status s = check_config(cfg, &d);
    if (s != STATEKV_OK) return s;
    if (!bytes) return STATEKV_ERR_INVALID_ARG;
    *bytes = make_layout(*cfg, d).total;
    return STATEKV_OK;
}

statekv_status statekv_init(const statekv_config* cfg, void* device_arena, size_t arena_bytes,
                            statekv_handle** out)
{
    Derived d;
    statekv_status s = check_config(cfg, &d);
    if (s != STATEKV_OK) return s;
    if (!out || !device_arena || !aligned(device_arena, kAlign)) return STATEKV_ERR_INVALID_ARG;
    const Layout lay = make_layout(*cfg, d);
    if (arena_bytes < lay.total) return STATEKV_ERR_ARENA_TOO_SMALL;
    if (!tma_encode_available()) return STATEKV_ERR_CUDA;

    statekv_handle* h = new (std::nothrow) statekv_handle();
    if (!h) return STATEKV_ERR_CUDA;
    h->cfg = *cfg;
    h->d = d;
    h->lay = lay;
    h->arena = static_cast<uint8_t*>(device_arena);
    h->frames_host.assign(static_cast<size_t>(d.SL), 0);
    h->text_host.assign(static_cast<size_t>(d.SL), 0);
    h->prof_on = false;
    h->prof_used = 0;
    std::memset(&h->tm_sk, 0, sizeof(CUtensorMap));
    std::memset(&h->tm_sv, 0, sizeof(CUtensorMap));
    std::memset(&h->tm_ck, 0, sizeof(CUtensorMap));
    std::memset(&h->tm_cv, 0, sizeof(CUtensorMap));
    std::memset(&h->tm_dk, 0, sizeof(CUtensorMap));
    std::memset(&h->tm_dv, 0, sizeof(CUtensorMap));

    void* st_host = nullptr;
    if (cudaHostAlloc(&st_host, 64, cudaHostAllocMapped) != cudaSuccess) {
        delete h;
        return STATEKV_ERR_CUDA;
    }
    h->status_host = static_cast<volatile int32_t*>(st_host);
    *h->status_host = 0;
    void* st_dev = nullptr;
    if (cudaHostGetDevicePointer(&st_dev, st_host, 0) != cudaSuccess) {
        cudaFreeHost(st_host);
        delete h;
        return STATEKV_ERR_CUDA;
    }
    h->status_dev = static_cast<int32_t*>(st_dev);

    const int D = cfg->head_dim, B = cfg->state_capacity, Hkv = cfg->num_kv_heads;
    bool ok = attn_prepare(D) == cudaSuccess && select_prepare() == cudaSuccess &&
              gemm_prepare() == cudaSuccess && thin_prepare() == cudaSuccess &&
              decode_prepare() == cudaSuccess;
    if (ok && B > 0) {
        const cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(B),
                                    static_cast<cuuint64_t>(Hkv), static_cast<cuuint64_t>(d.SL)};
        const cuuint64_t strides[3] = {static_cast<cuuint64_t>(D) * 2,
                                       static_cast<cuuint64_t>(B) * D * 2,
                                       static_cast<cuuint64_t>(Hkv) * B * D * 2};
        const cuuint32_t box[4] = {64, static_cast<cuuint32_t>(kBN), 1, 1};
        ok = encode_4d(&h->tm_sk, h->arena + lay.state_k, dims, strides, box) &&
             encode_4d(&h->tm_sv, h->arena + lay.state_v, dims, strides, box);
    }
    if (ok) {
        const cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(d.cap),
                                    static_cast<cuuint64_t>(Hkv), static_cast<cuuint64_t>(d.SL)};
        const cuuint64_t strides[3] = {static_cast<cuuint64_t>(D) * 2,
                                       static_cast<cuuint64_t>(d.cap) * D * 2,
                                       static_cast<cuuint64_t>(Hkv) * d.cap * D * 2};
        const cuuint32_t box[4] = {64, static_cast<cuuint32_t>(kBN), 1, 1};
        const cuuint32_t dbox[4] = {64, static_cast<cuuint32_t>(kDecodeKeyBox), 1, 1};
        ok = encode_4d(&h->tm_ck, h->arena + lay.cache_k, dims, strides, box) &&
             encode_4d(&h->tm_cv, h->arena + lay.cache_v, dims, strides, box) &&
             encode_4d(&h->tm_dk, h->arena + lay.cache_k, dims, strides, dbox) &&
             encode_4d(&h->tm_dv, h->arena + lay.cache_v, dims, strides, dbox);
    }
    ok = ok && create_streams(h);
    // Empty states and decode caches: zero rows, positions -1.  A key tile that
    // runs past the valid rows of a state or of the cache still reads them;
    // their scores are masked, but P = 0 times a non-finite value row would
    // still be NaN, so every row a tile can reach must hold finite values.
    ok = ok && cudaMemset(h->arena + lay.state_k, 0, lay.positions - lay.state_k) == cudaSuccess &&
         cudaMemset(h->arena + lay.positions, 0xFF, lay.counts - lay.positions) == cudaSuccess &&
         cudaMemset(h->arena + lay.counts, 0, lay.cache_k - lay.counts) == cudaSuccess &&
         cudaMemset(h->arena + lay.cache_k, 0, lay.partials - lay.cache_k) == cudaSuccess;
    for (int i = 0; ok && i < lay.guards.n; ++i)  // debug builds: the guard bands, after the fills above
        ok = cudaMemset(h->arena + lay.guards.off[i], kGuardFill, kGuard) == cudaSuccess;
    ok = ok && cudaDeviceSynchronize() == cudaSuccess;
    if (!ok) {
        cudaFreeHost(st_host);
        release_streams(h);
        delete h;
        return STATEKV_ERR_CUDA;
    }
    *out = h;
    return STATEKV_OK;
}

statekv_status statekv_prefill_frame(statekv_handle* h, const statekv_frame_args* args,
                                     statekv_stream stream)
{
    const statekv_status s = check_args(h, args, false);
    if (s != STATEKV_OK) return s;
    return run_step(h, *args, reinterpret_cast<cudaStream_t>(stream));
}

statekv_status statekv_debug_check(statekv_handle* h, statekv_stream stream)
{
    if (!h) return STATEKV_ERR_INVALID_ARG;
    if (!STATEKV_DEBUG_CHECKS) return STATEKV_ERR_UNSUPPORTED;
    if (*h->status_host != 0) return device_status(*h->status_host);
    return launch_canary_check(h->arena, h->lay.guards, h->status_dev,
                               reinterpret_cast<cudaStream_t>(stream)) == cudaSuccess
               ? STATEKV_OK
               : STATEKV_ERR_CUDA;
}

statekv_status statekv_full_attention_frame(statekv_handle* h, const statekv_frame_args* args,
                                           statekv_stream stream)
{
    const statekv_status s = check_args(h, args, false);
    if (s != STATEKV_OK) return s;
    if (args->importance) return STATEKV_ERR_INVALID_ARG;
    return run_full(h, *args, reinterpret_cast<cudaStream_t>(stream));
}

namespace {

// Columns of the attention kernel's partials in scores mode: every cache row
// (max_frames * T) then the frame's tokens.
long long scores_bp(const statekv_config& c)
{
    return static_cast<long long>(c.max_frames) * c.tokens_per_frame;
}

}  // namespace

statekv_status statekv_scores_workspace_bytes(const statekv_handle* h, int32_t stream_count,
                                              int32_t layer_count, size_t* bytes)
{
    if (!h || !bytes || stream_count < 1 || layer_count < 1 ||
        stream_count > h->cfg.num_streams || layer_count > h->cfg.num_layers)
        return STATEKV_ERR_INVALID_ARG;
    const long long pp = scores_bp(h->cfg) + h->cfg.tokens_per_frame;
    if (pp > 0x7FFFFFFFll) return STATEKV_ERR_UNSUPPORTED;
    *bytes = static_cast<size_t>(stream_count) * layer_count * h->cfg.num_kv_heads * h->d.MT *
             static_cast<size_t>(pp) * sizeof(float);
    return STATEKV_OK;
}

statekv_status statekv_full_attention_scores(statekv_handle* h, const statekv_frame_args* args,
                                             float* scores, void* workspace,
                                             size_t workspace_bytes, statekv_stream stream)
{
    const statekv_status s = check_args(h, args, false);
    if (s != STATEKV_OK) return s;
    if (args->importance || !scores || !workspace || !aligned(scores, 4) || !aligned(workspace, 16))
        return STATEKV_ERR_INVALID_ARG;
    size_t need = 0;
    const statekv_status w = statekv_scores_workspace_bytes(h, args->stream_count,
                                                            args->layer_count, &need);
    if (w != STATEKV_OK) return w;
    if (workspace_bytes < need) return STATEKV_ERR_INVALID_ARG;
    const statekv_config& c = h->cfg;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const long long bp = scores_bp(c);
    float* part = static_cast<float*>(workspace);
    const statekv_status r = run_full(h, *args, st, part, bp);
    if (r != STATEKV_OK) return r;
    ScoresParams sp{};
    sp.partials = part;
    sp.scores = scores;
    sp.frames = h->at<int32_t>(h->lay.frames);
    sp.units = UnitRange{args->stream_begin, args->layer_begin, args->layer_count, c.num_layers};
    sp.T = c.tokens_per_frame;
    sp.Hkv = c.num_kv_heads;
    sp.MT = h->d.MT;
    sp.Bp = bp;
    sp.Pp = bp + c.tokens_per_frame;
    sp.ncols = bp;
    if (launch_scores_reduce(sp, args->stream_count * args->layer_count, st) != cudaSuccess)
        return STATEKV_ERR_CUDA;
    return STATEKV_OK;
}

statekv_status statekv_topb_mask(const float* scores, int32_t rows, int64_t n, int64_t row_stride,
                                 int64_t B, uint8_t* mask, statekv_stream stream)
{
    if (!scores || !mask || !aligned(scores, 4) || rows < 0 || rows > 0x7FFFFFFF || n < 0 ||
        row_stride < n || row_stride > (1ll << 31) || B < 0)
        return STATEKV_ERR_INVALID_ARG;
    if (launch_topb_mask(scores, rows, n, row_stride, B, mask,
                         reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
        return STATEKV_ERR_CUDA;
    return STATEKV_OK;
}

statekv_status statekv_concentration_sums(const float* scores, const uint8_t* mask, int32_t rows,
                                          int64_t n, int64_t row_stride, double* out,
                                          statekv_stream stream)
{
    if (!scores || !mask || !out || !aligned(scores, 4) || !aligned(out, 8) || rows < 0 || n < 0 ||
        row_stride < n)
        return STATEKV_ERR_INVALID_ARG;
    if (launch_concentration(scores, mask, rows, n, row_stride, out,
                             reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
        return STATEKV_ERR_CUDA;
    return STATEKV_OK;
}

statekv_status statekv_state_metrics(const uint8_t* mask_n, const uint8_t* mask_n1,
                                     const float* scores_n1, int32_t rows, int64_t n_seen,
                                     int32_t T, int64_t row_stride, double* out,
                                     statekv_stream stream)
{
    if (!mask_n || !mask_n1 || !scores_n1 || !out || !aligned(scores_n1, 4) || !aligned(out, 8) ||
        rows < 0 || n_seen < 0 || T < 0 || n_seen + T > row_stride)
        return STATEKV_ERR_INVALID_ARG;
    if (launch_state_metrics(mask_n, mask_n1, scores_n1, rows, n_seen, T, row_stride, out,
                             reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
        return STATEKV_ERR_CUDA;
    return STATEKV_OK;
}

namespace {

// Workspace carve-up of one block call (all offsets 256-byte aligned).
struct BlockBufs {
    size_t h, qkv, q, k, v, attn, gu, act, rope, gemm_part, gemm_cnt, total;
};

// split-K tile counters: one region per projection GEMM of a block call (a
// split plan has fewer tiles than SMs), zeroed at the start of the call
constexpr int kGemmCounterRegion = 256;

// The four projection GEMMs of a layer at `rows` rows: (N, K) of QKV, O,
// gate/up and down.
void block_gemm_shapes(const statekv_config& c, const statekv_block_config& b, int (&nk)[4][2])
{
    const int d = c.head_dim, hq = c.num_q_heads, hkv = c.num_kv_heads;
    const int H = b.hidden, I = b.intermediate;
    nk[0][0] = (hq + 2 * hkv) * d;
    nk[0][1] = H;
    nk[1][0] = H;
    nk[1][1] = hq * d;
    nk[2][0] = 2 * I;
    nk[2][1] = H;
    nk[3][0] = H;
    nk[3][1] = I;
}

BlockBufs block_bufs(const statekv_config& c, const statekv_block_config& b, int streams)
{
    const size_t rows = static_cast<size_t>(streams) * c.tokens_per_frame;
    const size_t d = c.head_dim, hq = c.num_q_heads, hkv = c.num_kv_heads;
    auto up = [](size_t x) { return (x + 255) & ~static_cast<size_t>(255); };
    BlockBufs o{};
    size_t off = 0;
    auto take = [&](size_t bytes) {
        const size_t at = off;
        off += up(bytes);
        return at;
    };
    o.h = take(rows * b.hidden * 2);
    o.qkv = take(rows * (hq + 2 * hkv) * d * 2);
    o.q = take(rows * hq * d * 2);
    o.k = take(rows * hkv * d * 2);
    o.v = take(rows * hkv * d * 2);
    o.attn = take(rows * hq * d * 2);
    o.gu = take(rows * 2 * static_cast<size_t>(b.intermediate) * 2);
    o.act = take(rows * static_cast<size_t>(b.intermediate) * 2);
    o.rope = take(rows * (d / 2) * 8);  // (cos, sin) per row and rotated pair
    // split-K partials of the largest split GEMM, and the tile counters of
    // the cooperative path (rows above kThinMaxRows; the thin path adds its
    // splits up inside a thread-block cluster and needs neither)
    int nk[4][2];
    block_gemm_shapes(c, b, nk);
    size_t part = 0;
    const int sms = device_sm_count();
    if (rows > static_cast<size_t>(kThinMaxRows))
        for (int i = 0; i < 4; ++i)
            part = std::max(part, gemm_plan(static_cast<int>(rows), nk[i][0], nk[i][1], sms).partial_bytes);
    o.gemm_part = take(part);
    o.gemm_cnt = take(static_cast<size_t>(4) * c.num_layers * kGemmCounterRegion * 4);
    o.total = off;
    return o;
}

bool block_config_ok(const statekv_config& c, const statekv_block_config* b)
{
    return b && b->hidden > 0 && b->hidden % 8 == 0 && b->hidden <= 8192 && b->intermediate > 0 &&
           b->intermediate % 8 == 0 && b->rms_eps >= 0.f && std::isfinite(b->rms_eps) &&
           b->rope_theta > 1.f && std::isfinite(b->rope_theta) && std::isfinite(b->yarn_factor) &&
           (b->yarn_factor <= 1.f || b->yarn_original_max > 0) && c.head_dim / 2 <= 64;
}

}  // namespace

statekv_status statekv_block_workspace_bytes(const statekv_handle* h,
                                             const statekv_block_config* bc,
                                             int32_t stream_count, size_t* bytes)
{
    if (!h || !bytes || !block_config_ok(h->cfg, bc) || stream_count < 1 ||
        stream_count > h->cfg.num_streams)
        return STATEKV_ERR_INVALID_ARG;
    *bytes = block_bufs(h->cfg, *bc, stream_count).total;
    return STATEKV_OK;
}

statekv_status statekv_block_frame(statekv_handle* h, const statekv_block_config* bc,
                                   const statekv_block_weights* weights, int32_t stream_begin,
                                   int32_t stream_count, int32_t layer_begin, int32_t layer_count,
                                   const void* x_in, void* x_out, void* workspace,
                                   size_t workspace_bytes, statekv_stream stream)
{
    if (!h || !weights || !x_in || !x_out || !workspace || !block_config_ok(h->cfg, bc) ||
        !aligned(x_in, 16) || !aligned(x_out, 16) || !aligned(workspace, 256))
        return STATEKV_ERR_INVALID_ARG;
    const statekv_config& c = h->cfg;
    const statekv_block_config& b = *bc;
    if (stream_count < 1 || stream_begin < 0 || stream_begin + stream_count > c.num_streams ||
        layer_count < 1 || layer_begin < 0 || layer_begin + layer_count > c.num_layers)
        return STATEKV_ERR_INVALID_ARG;
    const BlockBufs bb = block_bufs(c, b, stream_count);
    if (workspace_bytes < bb.total) return STATEKV_ERR_INVALID_ARG;
    for (int l = layer_begin; l < layer_begin + layer_count; ++l) {
        const statekv_block_weights& w = weights[l];
        if (!w.norm_attn || !w.w_qkv || !w.w_o || !w.norm_mlp || !w.w_gate_up || !w.w_down ||
            !aligned(w.norm_attn, 16) || !aligned(w.w_qkv, 16) || !aligned(w.w_o, 16) ||
            !aligned(w.norm_mlp, 16) || !aligned(w.w_gate_up, 16) || !aligned(w.w_down, 16) ||
            (w.b_qkv && !aligned(w.b_qkv, 16)))
            return STATEKV_ERR_INVALID_ARG;
    }
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    auto buf = [&](size_t off) { return reinterpret_cast<__nv_bfloat16*>(ws + off); };
    // every covered (stream, layer) must be able to take the frame
    statekv_frame_args probe{};
    probe.stream_begin = stream_begin;
    probe.stream_count = stream_count;
    probe.layer_begin = layer_begin;
    probe.layer_count = layer_count;
    probe.q = buf(bb.q);
    probe.k = buf(bb.k);
    probe.v = buf(bb.v);
    probe.out = buf(bb.attn);
    const statekv_status s = check_args(h, &probe, false);
    if (s != STATEKV_OK) return s;

    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const int T = c.tokens_per_frame, d = c.head_dim, Hq = c.num_q_heads, Hkv = c.num_kv_heads;
    const int rows = stream_count * T;
    const int H = b.hidden, I = b.intermediate, W = (Hq + 2 * Hkv) * d;
    __nv_bfloat16* x = static_cast<__nv_bfloat16*>(x_out);
    if (x_out != x_in &&
        cudaMemcpyAsync(x, x_in, static_cast<size_t>(rows) * H * 2, cudaMemcpyDeviceToDevice,
                        st) != cudaSuccess)
        return STATEKV_ERR_CUDA;

    RopeParams rp{};
    rp.qkv = buf(bb.qkv);
    rp.q = buf(bb.q);
    rp.k = buf(bb.k);
    rp.v = buf(bb.v);
    rp.frames = h->at<int32_t>(h->lay.frames);
    rp.stream_begin = stream_begin;
    rp.num_layers = c.num_layers;
    rp.S = stream_count;
    rp.T = T;
    rp.Hq = Hq;
    rp.Hkv = Hkv;
    rp.d = d;
    {   // RoPE frequencies (fp64), with YaRN's blend when scaled
        const double pi2 = 6.283185307179586476925286766559;
        rp.scale = 1.f;
        for (int k = 0; k < d / 2; ++k) {
            double f = std::pow(static_cast<double>(b.rope_theta), -2.0 * k / d);
            if (b.yarn_factor > 1.f) {
                const double r = b.yarn_original_max * f / pi2;  // context / wavelength
                const double g = std::min(1.0, std::max(0.0, (r - 1.0) / 31.0));
                f = (1.0 - g) * f / b.yarn_factor + g * f;
            }
            rp.freq[k] = f;
        }
        if (b.yarn_factor > 1.f) rp.scale = static_cast<float>(0.1 * std::log(b.yarn_factor) + 1.0);
    }
    const int sms = device_sm_count();
    int* gemm_cnt = reinterpret_cast<int*>(ws + bb.gemm_cnt);
    if (cudaMemsetAsync(gemm_cnt, 0, static_cast<size_t>(4) * layer_count * kGemmCounterRegion * 4, st) !=
        cudaSuccess)
        return STATEKV_ERR_CUDA;
    int gemm_seq = 0;  // the call's projection GEMMs in order: each has its own counters
    // D[rows][N] = X[rows][K] W[N][K]^T (+ bias) (+ D), on the tensor cores
    // With pair_I > 0 (gate/up: N = 2 pair_I) and a plan without K split, D
    // receives SiLU(gate) * up [rows][pair_I] from the GEMM's epilogue and the
    // call returns 2; otherwise it returns 1 after storing the plain product.
    auto gemm = [&](const void* X, const void* Wt, const void* bias, __nv_bfloat16* D, bool add,
                    int N, int K, int pair_I = 0, __nv_bfloat16* D_pair = nullptr) -> int {
        const GemmPlan g = gemm_plan(rows, N, K, sms);
        if (g.counters > kGemmCounterRegion) return 0;
        const bool paired = pair_I > 0 && g.splits == 1;
        int* counters = gemm_cnt + static_cast<size_t>(gemm_seq++) * kGemmCounterRegion;
        CUtensorMap tx, tw;
        const cuuint64_t dx[4] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows), 1, 1};
        const cuuint64_t dw[4] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(paired ? pair_I : N),
                                  static_cast<cuuint64_t>(paired ? 2 : 1), 1};
        const cuuint64_t sx[3] = {static_cast<cuuint64_t>(K) * 2, static_cast<cuuint64_t>(K) * rows * 2,
                                  static_cast<cuuint64_t>(K) * rows * 2};
        const cuuint64_t sw[3] = {static_cast<cuuint64_t>(K) * 2,
                                  static_cast<cuuint64_t>(K) * (paired ? pair_I : N) * 2,
                                  static_cast<cuuint64_t>(K) * N * 2};
        const cuuint32_t box[4] = {static_cast<cuuint32_t>(kGemmBK), static_cast<cuuint32_t>(kGemmBM), 1, 1};
        const cuuint32_t wbox[4] = {static_cast<cuuint32_t>(kGemmBK),
                                    static_cast<cuuint32_t>(paired ? g.bn / 2 : g.bn), 1, 1};
        if (!encode_4d(&tx, X, dx, sx, box) || !encode_4d(&tw, Wt, dw, sw, wbox)) return false;
        GemmParams gp{};
        gp.M = rows;
        gp.N = paired ? pair_I : N;
        gp.K = K;
        gp.bn = g.bn;
        gp.paired_I = paired ? pair_I : 0;
        gp.n_tiles = paired ? (pair_I + g.bn / 2 - 1) / (g.bn / 2) : g.n_tiles;
        gp.k_steps = g.k_steps;
        gp.kps = g.kps;
        gp.splits = g.splits;
        gp.units = paired ? gp.n_tiles * g.m_pairs : g.units;
        gp.bias = static_cast<const __nv_bfloat16*>(bias);
        gp.D = paired ? D_pair : D;
        gp.add = add ? 1 : 0;
        gp.partials = reinterpret_cast<float*>(ws + bb.gemm_part);
        gp.counters = counters;
        gp.status = h->status_dev;
        gp.watchdog_ns = 1000000ull * (c.watchdog_ms ? c.watchdog_ms : 2000u);
        if (timed(h, 3, st, [&] { return launch_gemm(tx, tw, gp, sms, st); }) != cudaSuccess) return 0;
        return paired ? 2 : 1;
    };
    // Up to kThinMaxRows rows (one stream's frame) the projections run as thin
    // GEMMs whose epilogues finish the job: QKV adds the bias, rotates q and k
    // with the table the preceding RMSNorm wrote and stores q, k, v in the
    // step's layout; the output and down projections add into the residual
    // x; gate/up stores SiLU(gate) * up.
    const unsigned long long wd_ns = 1000000ull * (c.watchdog_ms ? c.watchdog_ms : 2000u);
    float2* rope_tab = reinterpret_cast<float2*>(ws + bb.rope);
    auto thin_gemm = [&](const void* X, const void* Wt, int Nw, int K, int paired_I, int op,
                         __nv_bfloat16* out, const void* bias) {
        const ThinPlan g = thin_plan(rows, Nw, K, sms, paired_I);
        CUtensorMap tx, tw;
        const cuuint64_t dx[4] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows), 1, 1};
        const cuuint64_t dw[4] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(Nw), 1, 1};
        const cuuint64_t sx[3] = {static_cast<cuuint64_t>(K) * 2, static_cast<cuuint64_t>(K) * rows * 2,
                                  static_cast<cuuint64_t>(K) * rows * 2};
        const cuuint64_t sw[3] = {static_cast<cuuint64_t>(K) * 2, static_cast<cuuint64_t>(K) * Nw * 2,
                                  static_cast<cuuint64_t>(K) * Nw * 2};
        const cuuint32_t bx[4] = {static_cast<cuuint32_t>(kGemmBK), static_cast<cuuint32_t>(g.Mp), 1, 1};
        const cuuint32_t bw[4] = {static_cast<cuuint32_t>(kGemmBK), 128, 1, 1};
        if (!encode_4d(&tx, X, dx, sx, bx) || !encode_4d(&tw, Wt, dw, sw, bw)) return false;
        ThinParams tp{};
        tp.M = rows;
        tp.Mp = g.Mp;
        tp.Nw = Nw;
        tp.K = K;
        tp.k_steps = g.k_steps;
        tp.kps = g.kps;
        tp.splits = g.splits;
        tp.stages = g.stages;
        tp.paired_I = paired_I;
        tp.wblocks = g.wblocks;
        tp.region = g.region;
        tp.op = op;
        tp.out = out;
        tp.bias = static_cast<const __nv_bfloat16*>(bias);
        tp.q = buf(bb.q);
        tp.k = buf(bb.k);
        tp.v = buf(bb.v);
        tp.rope = rope_tab;
        tp.Hq = Hq;
        tp.Hkv = Hkv;
        tp.d = d;
        tp.status = h->status_dev;
        tp.watchdog_ns = wd_ns;
        return timed(h, 3, st, [&] { return launch_thin_gemm(tx, tw, tp, g.smem, st); }) == cudaSuccess;
    };
    const bool thin = rows <= kThinMaxRows;
    for (int l = layer_begin; l < layer_begin + layer_count; ++l) {
        const statekv_block_weights& w = weights[l];
        rp.layer = l;
        if (thin) {
            // the norm also writes the rows' RoPE table for the QKV epilogue
            if (timed(h, 4, st, [&] {
                    return launch_rmsnorm_rope(x, static_cast<const __nv_bfloat16*>(w.norm_attn), b.rms_eps,
                                               buf(bb.h), rows, H, rp, rope_tab, st);
                }) != cudaSuccess ||
                !thin_gemm(buf(bb.h), w.w_qkv, W, H, 0, kThinQkvRope, nullptr, w.b_qkv))
                return STATEKV_ERR_CUDA;
        } else if (timed(h, 4, st, [&] {
                       return launch_rmsnorm(x, static_cast<const __nv_bfloat16*>(w.norm_attn), b.rms_eps,
                                             buf(bb.h), rows, H, st);
                   }) != cudaSuccess ||
                   !gemm(buf(bb.h), w.w_qkv, w.b_qkv, buf(bb.qkv), false, W, H) ||
                   timed(h, 4, st, [&] { return launch_qkv_rope(rp, st); }) != cudaSuccess) {
            return STATEKV_ERR_CUDA;
        }
        statekv_frame_args a = probe;
        a.layer_begin = l;
        a.layer_count = 1;
        const statekv_status r = run_step(h, a, st);
        if (r != STATEKV_OK) return r;
        if (thin) {
            if (!thin_gemm(buf(bb.attn), w.w_o, H, Hq * d, 0, kThinResidual, x, nullptr) ||
                timed(h, 4, st, [&] {
                    return launch_rmsnorm(x, static_cast<const __nv_bfloat16*>(w.norm_mlp), b.rms_eps,
                                          buf(bb.h), rows, H, st);
                }) != cudaSuccess ||
                !thin_gemm(buf(bb.h), w.w_gate_up, 2 * I, H, I, kThinSilu, buf(bb.act), nullptr) ||
                !thin_gemm(buf(bb.act), w.w_down, H, I, 0, kThinResidual, x, nullptr))
                return STATEKV_ERR_CUDA;
            continue;
        }
        if (!gemm(buf(bb.attn), w.w_o, nullptr, x, true, H, Hq * d)) return STATEKV_ERR_CUDA;
        if (timed(h, 4, st, [&] {
                return launch_rmsnorm(x, static_cast<const __nv_bfloat16*>(w.norm_mlp), b.rms_eps,
                                      buf(bb.h), rows, H, st);
            }) != cudaSuccess)
            return STATEKV_ERR_CUDA;
        // gate/up: SiLU(gate) * up in the GEMM's epilogue when its plan does not
        // split K, else the plain product and the elementwise kernel
        const int gu = gemm(buf(bb.h), w.w_gate_up, nullptr, buf(bb.gu), false, 2 * I, H, I, buf(bb.act));
        if (gu == 0) return STATEKV_ERR_CUDA;
        if (gu == 1 && timed(h, 4, st, [&] { return launch_silu_mul(buf(bb.gu), buf(bb.act), rows, I, st); }) !=
                           cudaSuccess)
            return STATEKV_ERR_CUDA;
        if (!gemm(buf(bb.act), w.w_down, nullptr, x, true, H, I)) return STATEKV_ERR_CUDA;
    }
    return STATEKV_OK;
}

statekv_status statekv_decode_step(statekv_handle* h, const statekv_decode_args* a,
                                  statekv_stream stream)
{
    if (!h || !a) return STATEKV_ERR_INVALID_ARG;
    const statekv_config& c = h->cfg;
    if (a->stream_count < 1 || a->layer_count < 1 || a->stream_begin < 0 || a->layer_begin < 0 ||
        a->stream_begin + a->stream_count > c.num_streams ||
        a->layer_begin + a->layer_count > c.num_layers || a->num_tokens < 1 ||
        a->num_tokens > kMaxFrameTokens)
        return STATEKV_ERR_INVALID_ARG;
    if (!a->q || !a->k || !a->v || !a->out || !aligned(a->q, 16) || !aligned(a->k, 16) ||
        !aligned(a->v, 16) || !aligned(a->out, 16))
        return STATEKV_ERR_INVALID_ARG;
    if (*h->status_host != 0) return device_status(*h->status_host);
    for (int s = a->stream_begin; s < a->stream_begin + a->stream_count; ++s)
        for (int l = a->layer_begin; l < a->layer_begin + a->layer_count; ++l) {
            const size_t unit = static_cast<size_t>(s) * c.num_layers + l;
            if (static_cast<long long>(h->frames_host[unit]) * c.tokens_per_frame +
                    h->text_host[unit] + a->num_tokens > h->d.cap)
                return STATEKV_ERR_CACHE_FULL;
        }
    return run_decode(h, *a, reinterpret_cast<cudaStream_t>(stream));
}

statekv_status statekv_prefill_frame_host(statekv_handle* h, const statekv_frame_args* args,
                                          statekv_stream stream)
{
    const statekv_status s = check_args(h, args, true);
    if (s != STATEKV_OK) return s;
    const statekv_config& c = h->cfg;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const size_t U = static_cast<size_t>(args->stream_count) * args->layer_count;
    const size_t T = c.tokens_per_frame, D = c.head_dim;
    const size_t qbytes = U * T * c.num_q_heads * D * 2;
    const size_t kvbytes = U * T * c.num_kv_heads * D * 2;
    const size_t impbytes = U * c.num_kv_heads * static_cast<size_t>(h->d.P) * 4;
    const Layout::Staging& g = h->lay.stg[0];
    statekv_frame_args dev = *args;
    dev.q = h->arena + g.q;
    dev.k = h->arena + g.k;
    dev.v = h->arena + g.v;
    dev.out = h->arena + g.out;
    dev.importance = args->importance ? h->at<float>(g.imp) : nullptr;
    // set 0 may still be in use by an earlier pipelined call
    if (cudaStreamWaitEvent(st, h->ev_comp[0], 0) != cudaSuccess ||
        cudaStreamWaitEvent(st, h->ev_out[0], 0) != cudaSuccess)
        return STATEKV_ERR_CUDA;
    if (cudaMemcpyAsync(const_cast<void*>(dev.q), args->q, qbytes, cudaMemcpyHostToDevice, st) !=
            cudaSuccess ||
        cudaMemcpyAsync(const_cast<void*>(dev.k), args->k, kvbytes, cudaMemcpyHostToDevice, st) !=
            cudaSuccess ||
        cudaMemcpyAsync(const_cast<void*>(dev.v), args->v, kvbytes, cudaMemcpyHostToDevice, st) !=
            cudaSuccess)
        return STATEKV_ERR_CUDA;
    const statekv_status r = run_step(h, dev, st);
    if (r != STATEKV_OK) return r;
    if (cudaMemcpyAsync(args->out, dev.out, qbytes, cudaMemcpyDeviceToHost, st) != cudaSuccess)
        return STATEKV_ERR_CUDA;
    if (args->importance &&
        cudaMemcpyAsync(args->importance, dev.importance, impbytes, cudaMemcpyDeviceToHost, st) !=
            cudaSuccess)
        return STATEKV_ERR_CUDA;
    return STATEKV_OK;
}

statekv_status statekv_prefill_frames_host(statekv_handle* h, const statekv_frame_args* frames,
                                           int32_t n, statekv_stream stream)
{
    if (!h || !frames || n < 1) return STATEKV_ERR_INVALID_ARG;
    const statekv_frame_args& f0 = frames[0];
    const statekv_status s = check_args(h, &f0, true);
    if (s != STATEKV_OK) return s;
    for (int32_t i = 1; i < n; ++i) {
        const statekv_frame_args& f = frames[i];
        if (f.stream_begin != f0.stream_begin || f.stream_count != f0.stream_count ||
            f.layer_begin != f0.layer_begin || f.layer_count != f0.layer_count || !f.q || !f.k ||
            !f.v || !f.out || (f.importance == nullptr) != (f0.importance == nullptr))
            return STATEKV_ERR_INVALID_ARG;
    }
    const statekv_config& c = h->cfg;
    for (int sI = f0.stream_begin; sI < f0.stream_begin + f0.stream_count; ++sI)
        for (int l = f0.layer_begin; l < f0.layer_begin + f0.layer_count; ++l)
            if (static_cast<long long>(h->frames_host[static_cast<size_t>(sI) * c.num_layers + l]) + n >
                c.max_frames)
                return STATEKV_ERR_CACHE_FULL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const size_t U = static_cast<size_t>(f0.stream_count) * f0.layer_count;
    const size_t T = c.tokens_per_frame, D = c.head_dim;
    const size_t qbytes = U * T * c.num_q_heads * D * 2;
    const size_t kvbytes = U * T * c.num_kv_heads * D * 2;
    const size_t impbytes = U * c.num_kv_heads * static_cast<size_t>(h->d.P) * 4;
    // the copies in start after the work already enqueued on the call's stream
    if (cudaEventRecord(h->ev_start, st) != cudaSuccess ||
        cudaStreamWaitEvent(h->cin, h->ev_start, 0) != cudaSuccess)
        return STATEKV_ERR_CUDA;
    for (int32_t i = 0; i < n; ++i) {
        const int b = i & 1;
        const Layout::Staging& g = h->lay.stg[b];
        const statekv_frame_args& f = frames[i];
        statekv_frame_args dev = f;
        dev.q = h->arena + g.q;
        dev.k = h->arena + g.k;
        dev.v = h->arena + g.v;
        dev.out = h->arena + g.out;
        dev.importance = f.importance ? h->at<float>(g.imp) : nullptr;
        // in: once the step that last read this staging set is done
        if (cudaStreamWaitEvent(h->cin, h->ev_comp[b], 0) != cudaSuccess ||
            cudaMemcpyAsync(const_cast<void*>(dev.q), f.q, qbytes, cudaMemcpyHostToDevice, h->cin) !=
                cudaSuccess ||
            cudaMemcpyAsync(const_cast<void*>(dev.k), f.k, kvbytes, cudaMemcpyHostToDevice, h->cin) !=
                cudaSuccess ||
            cudaMemcpyAsync(const_cast<void*>(dev.v), f.v, kvbytes, cudaMemcpyHostToDevice, h->cin) !=
                cudaSuccess ||
            cudaEventRecord(h->ev_in[b], h->cin) != cudaSuccess)
            return STATEKV_ERR_CUDA;
        // the step: after its inputs landed and the set's previous outputs left
        if (cudaStreamWaitEvent(st, h->ev_in[b], 0) != cudaSuccess ||
            cudaStreamWaitEvent(st, h->ev_out[b], 0) != cudaSuccess)
            return STATEKV_ERR_CUDA;
        const statekv_status r = run_step(h, dev, st);
        if (r != STATEKV_OK) return r;
        if (cudaEventRecord(h->ev_comp[b], st) != cudaSuccess ||
            cudaStreamWaitEvent(h->cout, h->ev_comp[b], 0) != cudaSuccess ||
            cudaMemcpyAsync(f.out, dev.out, qbytes, cudaMemcpyDeviceToHost, h->cout) != cudaSuccess ||
            (f.importance && cudaMemcpyAsync(f.importance, dev.importance, impbytes,
                                             cudaMemcpyDeviceToHost, h->cout) != cudaSuccess) ||
            cudaEventRecord(h->ev_out[b], h->cout) != cudaSuccess)
            return STATEKV_ERR_CUDA;
    }
    // later work on the call's stream sees every frame's results
    if (cudaStreamWaitEvent(st, h->ev_out[0], 0) != cudaSuccess ||
        cudaStreamWaitEvent(st, h->ev_out[1], 0) != cudaSuccess)
        return STATEKV_ERR_CUDA;
    return STATEKV_OK;
}

statekv_status statekv_watchdog_selftest(statekv_handle* h, statekv_stream stream)
{
    if (!h) return STATEKV_ERR_INVALID_ARG;
    const statekv_config& c = h->cfg;
    // One work unit (stream 0, layer 0) whose producer first waits on a barrier
    // that nothing completes: no input is read, no copy or MMA is issued, and
    // every role of the CTA leaves through its bounded waits.
    AttnParams pa{};
    pa.counts = h->at<int32_t>(h->lay.counts);
    pa.status = h->status_dev;
    pa.units = UnitRange{0, 0, 1, c.num_layers};
    pa.T = c.tokens_per_frame;
    pa.Hq = c.num_q_heads;
    pa.Hkv = c.num_kv_heads;
    pa.G = h->d.G;
    pa.B = c.state_capacity;
    pa.P = h->d.P;
    pa.MT = h->d.MT;
    pa.causal = c.causal_in_frame;
    pa.count_mul = 1;
    pa.scale_log2 = h->d.scale * 1.4426950408889634f;
    pa.watchdog_ns = 1000000ull * (c.watchdog_ms ? c.watchdog_ms : 2000u);
    pa.selftest_stall = 1;
    const cudaError_t e = launch_attn(c.head_dim, h->tm_sk, h->tm_sv, h->tm_sk, h->tm_sv, pa, 1,
                                      reinterpret_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? STATEKV_OK : STATEKV_ERR_CUDA;
}

statekv_status statekv_state_view(const statekv_handle* h, int32_t stream, int32_t layer,
                                  statekv_state_info* out)
{
    if (!h || !out || stream < 0 || layer < 0 || stream >= h->cfg.num_streams ||
        layer >= h->cfg.num_layers)
        return STATEKV_ERR_INVALID_ARG;
    const size_t unit = static_cast<size_t>(stream) * h->cfg.num_layers + layer;
    const size_t per = static_cast<size_t>(h->cfg.num_kv_heads) * h->cfg.state_capacity;
    out->k = h->arena + h->lay.state_k + unit * per * h->cfg.head_dim * 2;
    out->v = h->arena + h->lay.state_v + unit * per * h->cfg.head_dim * 2;
    out->positions = h->at<int32_t>(h->lay.positions) + unit * per;
    const int32_t f = h->frames_host[unit];
    const long long filled = static_cast<long long>(f) * h->cfg.tokens_per_frame;
    out->frames = f;
    out->count = static_cast<int32_t>(filled < h->cfg.state_capacity ? filled : h->cfg.state_capacity);
    out->virtual_len = filled;
    return STATEKV_OK;
}

statekv_status statekv_cache_view(const statekv_handle* h, int32_t stream, int32_t layer,
                                  statekv_cache_info* out)
{
    if (!h || !out || stream < 0 || layer < 0 || stream >= h->cfg.num_streams ||
        layer >= h->cfg.num_layers)
        return STATEKV_ERR_INVALID_ARG;
    const size_t unit = static_cast<size_t>(stream) * h->cfg.num_layers + layer;
    const size_t per = static_cast<size_t>(h->cfg.num_kv_heads) * h->d.cap * h->cfg.head_dim * 2;
    out->k = h->arena + h->lay.cache_k + unit * per;
    out->v = h->arena + h->lay.cache_v + unit * per;
    out->length = static_cast<int64_t>(h->frames_host[unit]) * h->cfg.tokens_per_frame +
                  h->text_host[unit];
    out->capacity = h->d.cap;
    return STATEKV_OK;
}

statekv_status statekv_profile_enable(statekv_handle* h, int32_t enable)
{
    if (!h) return STATEKV_ERR_INVALID_ARG;
    if (enable && h->prof.empty()) {
        h->prof.resize(kProfPairs);
        for (auto& r : h->prof)
            if (cudaEventCreate(&r.a) != cudaSuccess || cudaEventCreate(&r.b) != cudaSuccess)
                return STATEKV_ERR_CUDA;
    }
    if (enable) h->prof_used = 0;
    h->prof_on = enable != 0;
    return STATEKV_OK;
}

statekv_status statekv_profile_read(statekv_handle* h, statekv_profile* out)
{
    if (!h || !out) return STATEKV_ERR_INVALID_ARG;
    std::memset(out, 0, sizeof(*out));
    for (size_t i = 0; i < h->prof_used; ++i) {
        const ProfRec& r = h->prof[i];
        float ms = 0.f;
        if (cudaEventSynchronize(r.b) != cudaSuccess ||
            cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess)
            return STATEKV_ERR_CUDA;
        out->launches[r.kind] += 1;
        out->milliseconds[r.kind] += ms;
    }
    return STATEKV_OK;
}

statekv_status statekv_sync(statekv_handle* h)
{
    if (!h) return STATEKV_ERR_INVALID_ARG;
    if (cudaDeviceSynchronize() != cudaSuccess) return STATEKV_ERR_CUDA;
    return device_status(*h->status_host);
}

statekv_status statekv_device_error(const statekv_handle* h, int32_t* code)
{
    if (!h || !code) return STATEKV_ERR_INVALID_ARG;
    *code = *h->status_host;
    return STATEKV_OK;
}

void statekv_destroy(statekv_handle* h)
{
    if (!h) return;
    for (auto& r : h->prof) {
        cudaEventDestroy(r.a);
        cudaEventDestroy(r.b);
    }
    cudaFreeHost(const_cast<int32_t*>(h->status_host));
    release_streams(h);
    delete h;
}

const char* statekv_status_string(statekv_status s)
{
    switch (s) {
    case STATEKV_OK: return "ok";
    case STATEKV_ERR_INVALID_ARG: return "invalid argument";
    case STATEKV_ERR_UNSUPPORTED: return "unsupported configuration";
    case STATEKV_ERR_CACHE_FULL: return "decode cache full (max_frames reached)";
    case STATEKV_ERR_CUDA: return "CUDA runtime error";
    case STATEKV_ERR_DEVICE_TIMEOUT: return "device wait timed out";
    case STATEKV_ERR_ARENA_TOO_SMALL: return "arena too small";
    case STATEKV_ERR_DEVICE_FAULT: return "device-side consistency check failed";
    }
    return "unknown status";
}

}  // extern "C"
