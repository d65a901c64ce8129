// Decoding over the detailed cache (Sec. 3.2 / 3.3: decoding conditions on
// the detailed state D_N): a one-pass split-K attention for a few new tokens.
//
// Each of the n new tokens' G query heads of a KV head (R = n G <= 16 rows)
// attends to every cache row and, causally, to the new tokens, whose K/V rows
// the append kernel has already written after the cache's current length.
// Unlike the prefill kernel (two passes, so that the importance can use the
// final log-sum-exp), decoding needs no importance: one pass with an online
// max / sum per row streams each K and V row once.  The work is HBM-bound:
// at most 16 query rows meet each key, so the warp-level m16n8k16 MMA (rows
// padded to 16) keeps the instruction count far below the memory time.
//
//   decode_partial   grid (chunks, KV heads, units), 4 warps.  A warp takes 32
//                    keys at a time: their K and V rows arrive as TMA tensor
//                    copies (boxes of 64 columns x 32 keys of the cache's 4-D
//                    map, 128-byte swizzle), two steps ahead, into the warp's
//                    three-stage ring, each stage behind an mbarrier; fragment
//                    loads undo the swizzle, so they hit distinct banks.  Then
//                    S = Q K^T, the running max / sum per row, P in bf16,
//                    O += P V.  The 4 warps' (max, sum, O) merge into the
//                    chunk's partial.  Every wait is bounded by the watchdog.
//   decode_combine   one CTA per (unit, KV head): the chunks' partials merge
//                    (rescaled to the overall max) into O / sum, written as bf16.
#include "sm103_ptx.cuh"
#include "statekv_kernels.cuh"

namespace statekv {
namespace {

using namespace ptx;

constexpr int kDecThreads = 128;
constexpr int kDecWarps = kDecThreads / 32;
constexpr int kDecKeys = kDecodeKeyBox;  // keys per warp step (one TMA box)
constexpr int kDecStages = 3; // steps a warp has in flight or in use

template <int D>
struct DecLayout {
    // a 32-key tile of K (or V): D / 64 blocks of 32 rows x 128 bytes (64
    // columns), each in the TMA's 128-byte swizzle (1 KB atoms of 8 rows)
    static constexpr int kBlock = kDecKeys * 128;
    static constexpr int kMat = (D / 64) * kBlock;
    static constexpr int kStage = 2 * kMat;                  // K and V
    static constexpr int kWarp = kDecStages * kStage;
    static constexpr int kOffBar = kDecWarps * kWarp;        // full[warp][stage]
    static constexpr int kBytes = kOffBar + kDecWarps * kDecStages * 8;
    static constexpr int kAlloc = kBytes + 1024;             // room to align the base to 1 KB
    static_assert(kDecWarps * kDecodeRows * D * 4 + 2 * kDecWarps * kDecodeRows * 4 <= kOffBar,
                  "merge area fits");
    static_assert(kBlock % 1024 == 0, "swizzle atoms stay aligned");
};

// Byte offset of element (row, col) of a swizzled 32-key tile.
__device__ __forceinline__ uint32_t sw_off(int row, int col)
{
    const int blk = col >> 6, cc = col & 63;
    return blk * (kDecKeys * 128) + row * 128 + ((((cc >> 3) ^ (row & 7))) << 4) + ((cc & 7) << 1);
}

__device__ __forceinline__ unsigned long long dec_timer()
{
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ bool dec_wait(uint64_t* bar, uint32_t parity, unsigned long long deadline)
{
    for (;;) {
#pragma unroll 1
        for (int i = 0; i < 64; ++i)
            if (mbar_try_wait(bar, parity)) return true;
        if (dec_timer() > deadline) return false;
    }
}

__device__ __forceinline__ float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&h);
}

// D (16x8, fp32) += A (16x16 bf16, row) * B (16x8 bf16, col)
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7},"
        " {%8, %9}, {%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

template <int D>
__global__ void __launch_bounds__(kDecThreads)
    decode_partial(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                   const DecodeParams p)
{
    using L = DecLayout<D>;
    extern __shared__ uint8_t dsm_raw[];
    uint8_t* dsm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dsm_raw) + 1023) &
                                              ~static_cast<uintptr_t>(1023));
    const int chunk = blockIdx.x, hkv = blockIdx.y, u = blockIdx.z;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane >> 2, tig = lane & 3;  // fragment row group and column pair
    const int ua = p.units.unit_abs(u);
    const size_t head = static_cast<size_t>(ua) * p.Hkv + hkv;
    const int len0 = p.frames[head] * p.T + p.text[head];  // rows before the new tokens
    const int len = len0 + p.n;
    const int R = p.n * p.G;
    const int k0 = chunk * p.ck, k1 = min(len, k0 + p.ck);
    uint8_t* wsm = dsm + warp * L::kWarp;
    uint64_t* full = reinterpret_cast<uint64_t*>(dsm + L::kOffBar) + warp * kDecStages;
    if (lane == 0) {
        for (int s2 = 0; s2 < kDecStages; ++s2) mbar_init(&full[s2], 1);
        fence_mbar_init();
    }
    __syncwarp();
    const unsigned long long deadline = dec_timer() + p.watchdog_ns;
    bool ok = true;

    // Q as A fragments: row r = token r / G, head hkv G + r % G (rows >= R are 0)
    uint32_t qa[D / 16][4];
    {
        auto qval = [&](int r, int dd) -> float {
            if (r >= R) return 0.f;
            const int t = r / p.G, gg = r - t * p.G;
            return __bfloat162float(p.q[((static_cast<size_t>(u) * p.n + t) * p.Hq + hkv * p.G + gg) * D + dd]);
        };
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
            const int c = ks * 16 + 2 * tig;
            qa[ks][0] = pack_bf16(qval(g, c), qval(g, c + 1));
            qa[ks][1] = pack_bf16(qval(g + 8, c), qval(g + 8, c + 1));
            qa[ks][2] = pack_bf16(qval(g, c + 8), qval(g, c + 9));
            qa[ks][3] = pack_bf16(qval(g + 8, c + 8), qval(g + 8, c + 9));
        }
    }
    // the 32 K and V rows from key `base` into stage st, by one lane (rows past
    // the cache capacity read as zero; their scores are masked)
    auto load_step = [&](int base, int st) {
        if (lane == 0) {
            uint8_t* ks = wsm + st * L::kStage;
            uint8_t* vs = ks + L::kMat;
            fence_proxy_async_smem();  // the warp's earlier reads of this stage come first
            mbar_arrive_expect_tx(&full[st], 2 * L::kMat);
#pragma unroll
            for (int hb = 0; hb < D / 64; ++hb) {
                tma_load_4d(ks + hb * L::kBlock, &tm_k, &full[st], hb * 64, base, hkv, ua);
                tma_load_4d(vs + hb * L::kBlock, &tm_v, &full[st], hb * 64, base, hkv, ua);
            }
        }
    };

    const float c = p.scale_log2;
    float m[2] = {-INFINITY, -INFINITY}, l[2] = {0.f, 0.f};  // rows g and g + 8
    float o[D / 8][4];
#pragma unroll
    for (int nd = 0; nd < D / 8; ++nd)
#pragma unroll
        for (int e = 0; e < 4; ++e) o[nd][e] = 0.f;

    const int stride = kDecWarps * kDecKeys;
    const int base0 = k0 + warp * kDecKeys;
    const int nsteps = base0 < k1 ? (k1 - base0 + stride - 1) / stride : 0;
    // kDecStages - 1 steps ahead
#pragma unroll
    for (int s0 = 0; s0 < kDecStages - 1; ++s0)
        if (s0 < nsteps) load_step(base0 + s0 * stride, s0);
    int step = 0;
    for (; step < nsteps; ++step) {
        const int base = base0 + step * stride;
        const int st = step % kDecStages;
        const int pre = step + kDecStages - 1;
        // the stage `pre` lands in was read by step - 1, which this warp finished
        if (pre < nsteps) load_step(base0 + pre * stride, pre % kDecStages);
        ok = __all_sync(0xffffffffu, dec_wait(&full[st], (step / kDecStages) & 1, deadline));
        if (!ok) break;
        const uint8_t* ks = wsm + st * L::kStage;
        const uint8_t* vs = ks + L::kMat;
        // S = Q K^T: 4 key tiles of 8
        float sc[4][4];
#pragma unroll
        for (int nt = 0; nt < 4; ++nt) {
#pragma unroll
            for (int e = 0; e < 4; ++e) sc[nt][e] = 0.f;
#pragma unroll
            for (int kst = 0; kst < D / 16; ++kst) {
                const int kr = nt * 8 + g, kc = kst * 16 + 2 * tig;
                mma16816(sc[nt], qa[kst], *reinterpret_cast<const uint32_t*>(ks + sw_off(kr, kc)),
                         *reinterpret_cast<const uint32_t*>(ks + sw_off(kr, kc + 8)));
            }
        }
        // masks, running max / sum of rows g (h = 0) and g + 8 (h = 1)
        float alpha[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int r = g + 8 * h;
            const int lim = r < R ? min(k1, len0 + r / p.G + 1) : 0;  // keys [.., lim) visible
            float mx = -INFINITY;
#pragma unroll
            for (int nt = 0; nt < 4; ++nt)
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const int key = base + nt * 8 + 2 * tig + e;
                    float& v = sc[nt][2 * h + e];
                    v = key < lim ? v * c : -INFINITY;
                    mx = fmaxf(mx, v);
                }
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
            const float mn = fmaxf(m[h], mx);
            alpha[h] = mn == -INFINITY ? 1.f : ex2(m[h] - mn);
            float sum = 0.f;
#pragma unroll
            for (int nt = 0; nt < 4; ++nt)
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    float& v = sc[nt][2 * h + e];
                    v = mn == -INFINITY ? 0.f : ex2(v - mn);
                    sum += v;
                }
            sum += __shfl_xor_sync(0xffffffffu, sum, 1);
            sum += __shfl_xor_sync(0xffffffffu, sum, 2);
            l[h] = l[h] * alpha[h] + sum;
            m[h] = mn;
        }
#pragma unroll
        for (int nd = 0; nd < D / 8; ++nd) {
            o[nd][0] *= alpha[0];
            o[nd][1] *= alpha[0];
            o[nd][2] *= alpha[1];
            o[nd][3] *= alpha[1];
        }
        // O += P V: P as A fragments (keys 16j .. 16j + 15 are tiles 2j, 2j + 1)
#pragma unroll
        for (int j = 0; j < 2; ++j) {
            const uint32_t pa[4] = {pack_bf16(sc[2 * j][0], sc[2 * j][1]),
                                    pack_bf16(sc[2 * j][2], sc[2 * j][3]),
                                    pack_bf16(sc[2 * j + 1][0], sc[2 * j + 1][1]),
                                    pack_bf16(sc[2 * j + 1][2], sc[2 * j + 1][3])};
            const int vr0 = 16 * j + 2 * tig;
#pragma unroll
            for (int nd = 0; nd < D / 8; ++nd) {
                const int vc = nd * 8 + g;
                auto vat = [&](int r) { return *reinterpret_cast<const __nv_bfloat16*>(vs + sw_off(r, vc)); };
                __nv_bfloat162 b0, b1;
                b0.x = vat(vr0);
                b0.y = vat(vr0 + 1);
                b1.x = vat(vr0 + 8);
                b1.y = vat(vr0 + 9);
                mma16816(o[nd], pa, *reinterpret_cast<const uint32_t*>(&b0),
                         *reinterpret_cast<const uint32_t*>(&b1));
            }
        }
        __syncwarp();  // the stage is refilled kDecStages - 1 steps later
    }
    if (!ok) {
        if (lane == 0) *reinterpret_cast<volatile int32_t*>(p.status) = DEV_TIMEOUT_DECODE;
        // let the copies already issued land before the shared memory is reused
        if (lane == 0)
            for (int s2 = step; s2 < min(nsteps, step + kDecStages); ++s2)
                dec_wait(&full[s2 % kDecStages], (s2 / kDecStages) & 1, dec_timer() + p.watchdog_ns);
    }
    __syncthreads();

    // merge the 4 warps into the chunk's partial (reusing the staging memory)
    float* mo = reinterpret_cast<float*>(dsm);                       // [warp][16][D]
    float* mm = mo + kDecWarps * kDecodeRows * D;                     // [warp][16]
    float* ml = mm + kDecWarps * kDecodeRows;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int r = g + 8 * h;
        if (tig == 0) {
            mm[warp * kDecodeRows + r] = m[h];
            ml[warp * kDecodeRows + r] = l[h];
        }
#pragma unroll
        for (int nd = 0; nd < D / 8; ++nd) {
            mo[(warp * kDecodeRows + r) * D + nd * 8 + 2 * tig] = o[nd][2 * h];
            mo[(warp * kDecodeRows + r) * D + nd * 8 + 2 * tig + 1] = o[nd][2 * h + 1];
        }
    }
    __syncthreads();
    const size_t pidx = (static_cast<size_t>(u) * p.Hkv + hkv) * p.nchunk + chunk;
    float* po = p.part_o + pidx * kDecodeRows * D;
    float* pml = p.part_ml + pidx * kDecodeRows * 2;
    for (int i = threadIdx.x; i < R * D; i += kDecThreads) {
        const int r = i / D, dd = i - r * D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < kDecWarps; ++w) M = fmaxf(M, mm[w * kDecodeRows + r]);
        float ov = 0.f, Lv = 0.f;
        if (M != -INFINITY) {
#pragma unroll
            for (int w = 0; w < kDecWarps; ++w) {
                const float mw = mm[w * kDecodeRows + r];
                const float f = mw == -INFINITY ? 0.f : ex2(mw - M);
                ov += mo[(w * kDecodeRows + r) * D + dd] * f;
                Lv += ml[w * kDecodeRows + r] * f;
            }
        }
        po[r * D + dd] = ov;
        if (dd == 0) {
            pml[2 * r] = M;
            pml[2 * r + 1] = Lv;
        }
    }
}

// One CTA per (unit, KV head): O = sum_c O_c 2^(m_c - M) / sum_c l_c 2^(m_c - M).
template <int D>
__global__ void __launch_bounds__(256) decode_combine(const DecodeParams p)
{
    const int hkv = blockIdx.x, u = blockIdx.y;
    const int R = p.n * p.G;
    const size_t pbase = (static_cast<size_t>(u) * p.Hkv + hkv) * p.nchunk;
    for (int i = threadIdx.x; i < R * D; i += 256) {
        const int r = i / D, dd = i - r * D;
        float M = -INFINITY;
        for (int ch = 0; ch < p.nchunk; ++ch) M = fmaxf(M, p.part_ml[((pbase + ch) * kDecodeRows + r) * 2]);
        float o = 0.f, L = 0.f;
        for (int ch = 0; ch < p.nchunk; ++ch) {
            const float mc = p.part_ml[((pbase + ch) * kDecodeRows + r) * 2];
            if (mc == -INFINITY) continue;
            const float f = ex2(mc - M);
            L += p.part_ml[((pbase + ch) * kDecodeRows + r) * 2 + 1] * f;
            o += p.part_o[((pbase + ch) * kDecodeRows + r) * D + dd] * f;
        }
        const int t = r / p.G, g = r - t * p.G;
        p.out[((static_cast<size_t>(u) * p.n + t) * p.Hq + hkv * p.G + g) * D + dd] =
            __float2bfloat16(o / L);
    }
}

}  // namespace

cudaError_t launch_decode(const CUtensorMap& tm_k, const CUtensorMap& tm_v, const DecodeParams& p, int D,
                          int U, cudaStream_t st)
{
    if (U <= 0) return cudaSuccess;
    const dim3 g1(p.nchunk, p.Hkv, U), g2(p.Hkv, U);
    if (D == 64) {
        decode_partial<64><<<g1, kDecThreads, DecLayout<64>::kAlloc, st>>>(tm_k, tm_v, p);
        decode_combine<64><<<g2, 256, 0, st>>>(p);
    } else {
        decode_partial<128><<<g1, kDecThreads, DecLayout<128>::kAlloc, st>>>(tm_k, tm_v, p);
        decode_combine<128><<<g2, 256, 0, st>>>(p);
    }
    return cudaGetLastError();
}

cudaError_t decode_prepare()
{
    cudaError_t e = cudaFuncSetAttribute(decode_partial<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         DecLayout<64>::kAlloc);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(decode_partial<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                DecLayout<128>::kAlloc);
}

}  // namespace statekv
