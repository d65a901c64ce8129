// Projection GEMMs of the per-frame transformer block on the 5th-generation
// tensor cores:  D[M][N] = X[M][K] W[N][K]^T (+ bias[N]) (+ D when add), bf16
// in and out, fp32 accumulation in TMEM.
//
// X holds the block's activations (M = streams x tokens rows), W one weight
// matrix in the torch.nn.Linear layout [out][in].  At one stream M = 196, so
// every weight element is used by few rows and the product streams W from HBM;
// the kernel is built to read each weight byte once:
//   - a work unit is one 128-column tile of W (and of D) for a pair of 128-row
//     tiles of X (both accumulators live in TMEM, so a W tile is loaded once
//     for up to 256 rows), over one contiguous range of K;
//   - when the (column tile, row pair) grid alone would leave SMs idle, K is
//     split into ranges: every split writes an fp32 partial of its tile; the
//     launch is cooperative, so the splits of a tile wait for one another (an
//     atomic counter per tile, bounded by the watchdog), then split s adds its
//     share of the rows over every split in split order, so the result does
//     not depend on timing;
//   - one CTA per SM walks the units; TMEM holds two accumulator sets, so the
//     epilogue of one unit overlaps the main loop of the next;
//   - GEMMs whose 128-wide tiles would take several rounds on the SMs use W
//     tiles of 192 or 256 rows when fewer rounds of those cost less (every
//     projection at eight streams, gate/up from two): one accumulator set, and
//     each staged byte feeds up to 1.5x the MMA work.
// 192 threads: warp 0 issues the TMA loads (a four-stage ring of 48 KB: X rows
// m0..m0+127, X rows m0+128..m0+255, W rows n0..n0+127, 64 K-columns each,
// 128-byte swizzle), warp 1 allocates TMEM and issues tcgen05.mma
// (128 x 128 x 16, both operands K-major in shared memory), warps 2..5 read
// the accumulators (one TMEM lane quadrant each, thread = row) and write D or
// the fp32 partials.  Every mbarrier wait is bounded by the watchdog; on
// expiry the CTA records DEV_TIMEOUT_GEMM, drains and exits.
#include <algorithm>

#include "sm103_ptx.cuh"
#include "statekv_kernels.cuh"

namespace statekv {
namespace {

using namespace ptx;

constexpr int kGThreads = 192;
constexpr int kGTileA = kGemmBM * kGemmBK * 2;        // 16 KB: 128 rows of X x 64 K
// epilogue staging: per epilogue warp a 32 x 36 fp32 block (row-major, 16-byte
// rows padded by one float4 against bank conflicts) turns thread-per-row TMEM
// reads into row-contiguous global stores
constexpr int kGStageLd = 36;
constexpr int kRG = 8;  // rows per group of the split-K reduction (2 kRG loads in flight)

// Shared memory and TMEM plan for a tile of 256 rows of X x BN rows of W.
// BN = 128: a four-stage ring of 48 KB and two accumulator sets (2 x 128
// TMEM columns each), so a unit's epilogue overlaps the next unit's main loop.
// BN = 192 / 256: a three-stage ring of 56 / 64 KB and one set, its two
// 128-row accumulators at TMEM columns 0 and 256; each byte staged feeds up to
// 1.5x the MMA work of BN = 128, and the wider tiles change how many rounds a
// GEMM's tiles take on the SMs.
template <int BN>
struct GLayout {
    static constexpr int kStages = BN == 128 ? 4 : 3;
    static constexpr int kAccSets = BN == 128 ? 2 : 1;
    static constexpr int kMtStride = BN == 128 ? 128 : 256;  // TMEM columns between the two row tiles
    static constexpr int kSetStride = 256;                   // TMEM columns between accumulator sets
    static constexpr int kTileB = BN * kGemmBK * 2;
    static constexpr int kStageBytes = 2 * kGTileA + kTileB;
    static constexpr int kOffEpi = kStages * kStageBytes;
    static constexpr int kOffBar = kOffEpi + 4 * 32 * kGStageLd * 4;
    static constexpr int kNumBars = 2 * kStages + 5;  // full[S] empty[S] acc_full[2] acc_empty[2] drain
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;
    static constexpr int kBytes = kOffMisc + 16;
    static constexpr int kAlloc = kBytes + 1024;      // room to align the base to 1 KB
    // the epilogue reads the accumulators in 32-column chunks (paired: 32 gate and 32 up
    // columns at a time), so BN is a multiple of 64
    static_assert(BN == 128 || BN == 192 || BN == 256, "tile width");
    static_assert((kAccSets - 1) * kSetStride + kMtStride + BN <= 512, "TMEM columns");
    static_assert(kAlloc <= 232448, "shared memory budget");
    static_assert(kStageBytes % 1024 == 0 && kGTileA % 1024 == 0, "swizzle atoms stay aligned");
};

__device__ __forceinline__ unsigned long long g_globaltimer()
{
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ bool g_wait(uint64_t* bar, uint32_t parity, unsigned long long deadline)
{
    for (;;) {
#pragma unroll 1
        for (int i = 0; i < 64; ++i)
            if (mbar_try_wait(bar, parity)) return true;
        if (g_globaltimer() > deadline) return false;
    }
}

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

struct GemmUnit {
    int tile, split, n0, m0, ks0, ks1;
    bool two;  // the pair's second 128-row tile holds rows below M
};

// SiLU(g) * u with the fast exponential and division: straight-line code the
// compiler interleaves across a thread's 32 values (the epilogue runs one
// warp per SM sub-partition, so it is bound by dependent-instruction latency;
// the library expf / IEEE division branch and serialise it).  Relative error
// ~1e-6, far below the bf16 rounding of the result.
__device__ __forceinline__ float silu_times(float g, float u) { return __fdividef(g, 1.f + __expf(-g)) * u; }

// Round-to-nearest-even to bf16 of a finite float, as integer arithmetic on
// its bits (full-rate ALU work, where the conversion instructions are not):
// the same result as __float2bfloat16_rn for every finite input.
__device__ __forceinline__ uint32_t bf16_rne_bits(float x)
{
    const uint32_t u = __float_as_uint(x);
    return (u + 0x7FFFu + ((u >> 16) & 1u)) >> 16;
}

__device__ __forceinline__ float bf16_round(float x) { return __uint_as_float(bf16_rne_bits(x) << 16); }

// Tiles are numbered row pair fastest: the CTAs running at the same time
// share W tiles (each W tile is read from HBM about once and served from L2 to
// its other row pairs) while the X rows, far smaller, stay in L2.  Numbered
// column fastest, a GEMM whose W exceeds L2 re-read it from HBM once per row
// pair (1.94 GB of DRAM traffic for the 0.34 GB of the 8-stream gate/up).
template <int BN>
__device__ __forceinline__ GemmUnit gemm_unit(const GemmParams& p, int w)
{
    GemmUnit x;
    x.tile = w / p.splits;
    x.split = w - x.tile * p.splits;
    const int m_pairs = (p.M + 2 * kGemmBM - 1) / (2 * kGemmBM);
    x.n0 = (x.tile / m_pairs) * (p.paired_I ? BN / 2 : BN);  // paired: the output column base
    x.m0 = (x.tile % m_pairs) * 2 * kGemmBM;
    x.ks0 = x.split * p.kps;
    x.ks1 = min(p.k_steps, x.ks0 + p.kps);
    x.two = x.m0 + kGemmBM < p.M;
    return x;
}

// One element of D: bf16(acc + bias[n] (+ D[m][n])).  Lanes of a warp take
// consecutive n, so the loads and stores are row-contiguous.
__device__ __forceinline__ void store_elem(const GemmParams& p, int m, int n, float acc, float bias)
{
    if (m >= p.M || n >= p.N) return;
    __nv_bfloat16* dst = p.D + static_cast<size_t>(m) * p.N + n;
    float f = acc + bias;
    if (p.add) f += __bfloat162float(*dst);
    *dst = __float2bfloat16_rn(f);
}

// 4 consecutive columns n..n+3 of D, adding the residual when p.add.  The
// residual loads of every row are in flight before any store.
template <int NR>
__device__ __forceinline__ void store4_rows(const GemmParams& p, int m0, int mstep, int nrows, int n,
                                            float4 (&a)[NR])
{
    if (n >= p.N) return;
    if (n + 4 <= p.N && (p.N & 3) == 0) {
        if (p.add) {
            uint2 old[NR];
#pragma unroll
            for (int i = 0; i < NR; ++i)
                if (i < nrows) old[i] = *reinterpret_cast<const uint2*>(p.D + static_cast<size_t>(m0 + i * mstep) * p.N + n);
#pragma unroll
            for (int i = 0; i < NR; ++i)
                if (i < nrows) {
                    const __nv_bfloat162* o2 = reinterpret_cast<const __nv_bfloat162*>(&old[i]);
                    const float2 lo = __bfloat1622float2(o2[0]), hi = __bfloat1622float2(o2[1]);
                    a[i].x += lo.x;
                    a[i].y += lo.y;
                    a[i].z += hi.x;
                    a[i].w += hi.y;
                }
        }
#pragma unroll
        for (int i = 0; i < NR; ++i)
            if (i < nrows)
                *reinterpret_cast<uint2*>(p.D + static_cast<size_t>(m0 + i * mstep) * p.N + n) =
                    make_uint2(pack_bf16x2(a[i].x, a[i].y), pack_bf16x2(a[i].z, a[i].w));
    } else {
        for (int i = 0; i < nrows; ++i) {
            const int m = m0 + i * mstep;
            store_elem(p, m, n, a[i].x, 0.f);
            store_elem(p, m, n + 1, a[i].y, 0.f);
            store_elem(p, m, n + 2, a[i].z, 0.f);
            store_elem(p, m, n + 3, a[i].w, 0.f);
        }
    }
}

// Rows mrow0 + 4 q + sub (q < 8, below rmax) of one 32-column chunk, columns
// n..n+3, plus bias.
__device__ __forceinline__ void store_rows4(const GemmParams& p, int mrow0, int sub, int rmax, int n,
                                            float4 (&acc)[8])
{
    if (n >= p.N) return;
    float b[4] = {0.f, 0.f, 0.f, 0.f};
    if (p.bias)
#pragma unroll
        for (int e = 0; e < 4; ++e) b[e] = n + e < p.N ? __bfloat162float(p.bias[n + e]) : 0.f;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        acc[q].x += b[0];
        acc[q].y += b[1];
        acc[q].z += b[2];
        acc[q].w += b[3];
    }
    const int nrows = rmax > sub ? (rmax - sub + 3) / 4 : 0;  // rows 4 q + sub < rmax
    store4_rows<8>(p, mrow0 + sub, 4, nrows < 8 ? nrows : 8, n, acc);
}

template <int NR>
__device__ __forceinline__ void store_rows_strided(const GemmParams& p, int m0, int mstep, int nrows,
                                                   int n, float4 (&a)[NR])
{
    store4_rows<NR>(p, m0, mstep, nrows, n, a);
}

template <int BN>
__global__ void __launch_bounds__(kGThreads, 1)
    gemm_bf16_tc(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_w,
                 const GemmParams p)
{
    using L = GLayout<BN>;
    constexpr int kGStages = L::kStages, kGStageBytes = L::kStageBytes, kGTileB = L::kTileB;
    constexpr int NB = L::kAccSets;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + L::kOffBar);
    uint64_t* full = bars;                     // stage loaded
    uint64_t* empty = bars + kGStages;         // stage read by its MMAs
    uint64_t* acc_full = bars + 2 * kGStages;  // accumulator set complete
    uint64_t* acc_empty = acc_full + 2;        // accumulator set read out
    uint64_t* drain = acc_full + 4;            // every MMA of the CTA has completed
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + L::kOffMisc);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(sm + L::kOffMisc + 4);
    volatile int* last_flag = reinterpret_cast<volatile int*>(sm + L::kOffMisc + 8);
    const bool split = BN == 128 && p.splits > 1;  // the plan splits K only with 128-wide tiles

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int i = 0; i < kGStages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], 128);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, 512);
        tmem_relinquish();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tmem_slot;
    auto fail = [&](int site) {
        if (atomicExch(const_cast<int*>(abort_flag), 1) == 0)
            *reinterpret_cast<volatile int32_t*>(p.status) = DEV_TIMEOUT_GEMM | (site << 8);
    };

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            tma_prefetch_desc(&tm_x);
            tma_prefetch_desc(&tm_w);
            int last_use[kGStages];
#pragma unroll
            for (int s = 0; s < kGStages; ++s) last_use[s] = -1;
            bool ok = true;
            int n = 0;
            for (int w = blockIdx.x; ok && w < p.units; w += gridDim.x) {
                const GemmUnit x = gemm_unit<BN>(p, w);
                const unsigned long long deadline = g_globaltimer() + p.watchdog_ns;
                for (int ks = x.ks0; ks < x.ks1; ++ks, ++n) {
                    if (*abort_flag) {
                        ok = false;
                        break;
                    }
                    const int s = n % kGStages, use = n / kGStages;
                    if (use >= 1 && !g_wait(&empty[s], (use - 1) & 1, deadline)) {
                        fail(2);
                        ok = false;
                        break;
                    }
                    uint8_t* base = sm + s * kGStageBytes;
                    mbar_arrive_expect_tx(&full[s], (x.two ? 2 : 1) * kGTileA + kGTileB);
                    const int kc = ks * kGemmBK;
                    tma_load_4d(base, &tm_x, &full[s], kc, x.m0, 0, 0);
                    if (x.two) tma_load_4d(base + kGTileA, &tm_x, &full[s], kc, x.m0 + kGemmBM, 0, 0);
                    if (p.paired_I) {  // BN / 2 gate rows, then the same up rows
                        tma_load_4d(base + 2 * kGTileA, &tm_w, &full[s], kc, x.n0, 0, 0);
                        tma_load_4d(base + 2 * kGTileA + kGTileB / 2, &tm_w, &full[s], kc, x.n0, 1, 0);
                    } else {
                        tma_load_4d(base + 2 * kGTileA, &tm_w, &full[s], kc, x.n0, 0, 0);
                    }
                    last_use[s] = use;
                }
            }
            // let every copy land before the CTA's memory goes away
            const unsigned long long dl = g_globaltimer() + p.watchdog_ns;
            for (int s = 0; s < kGStages; ++s)
                if (last_use[s] >= 0) g_wait(&full[s], last_use[s] & 1, dl);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t kId = idesc_bf16_f32(kGemmBM, BN, false, false);
            const uint32_t s0 = smem_addr(sm);
            bool ok = true;
            int n = 0, u = 0, site = 3;
            for (int w = blockIdx.x; ok && w < p.units; w += gridDim.x, ++u) {
                const GemmUnit x = gemm_unit<BN>(p, w);
                const unsigned long long deadline = g_globaltimer() + p.watchdog_ns;
                const int buf = u % NB;
                site = 4;
                if (u >= NB && !(ok = g_wait(&acc_empty[buf], ((u - NB) / NB) & 1, deadline))) break;
                tc_fence_after();
                const uint32_t acc0 = tbase + buf * L::kSetStride, acc1 = acc0 + L::kMtStride;
                for (int ks = x.ks0; ks < x.ks1; ++ks, ++n) {
                    const int s = n % kGStages;
                    site = 3;
                    if (!(ok = g_wait(&full[s], (n / kGStages) & 1, deadline))) break;
                    tc_fence_after();
                    const uint32_t sa = s0 + s * kGStageBytes;
                    const uint64_t da0 = sdesc_sw128(sa, 16, 1024);
                    const uint64_t da1 = sdesc_sw128(sa + kGTileA, 16, 1024);
                    const uint64_t db = sdesc_sw128(sa + 2 * kGTileA, 16, 1024);
#pragma unroll
                    for (int kk = 0; kk < kGemmBK / 16; ++kk) {
                        // 16 K-elements = 32 bytes further along each 128-byte row
                        const uint32_t acc = (ks > x.ks0 || kk > 0) ? 1u : 0u;
                        umma_bf16(acc0, da0 + 2 * kk, db + 2 * kk, kId, acc);
                        if (x.two) umma_bf16(acc1, da1 + 2 * kk, db + 2 * kk, kId, acc);
                    }
                    umma_commit(&empty[s]);
                }
                if (!ok) break;
                umma_commit(&acc_full[buf]);
            }
            if (!ok) fail(site);
            // every MMA issued so far must finish before TMEM is released
            umma_commit(drain);
            g_wait(drain, 0, g_globaltimer() + p.watchdog_ns);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue (warps 2..5)
        const int quad = warp & 3;  // TMEM lane quadrant: rows 32 quad .. 32 quad + 31 of a tile
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        float* stg = reinterpret_cast<float*>(sm + L::kOffEpi) + (warp - 2) * 32 * kGStageLd;
        const int sub = lane >> 3, c4 = lane & 7;  // staging read-out: 4 rows x 8 float4 per instruction
        bool ok = true;
        int u = 0;
        for (int w = blockIdx.x; w < p.units; w += gridDim.x, ++u) {
            const GemmUnit x = gemm_unit<BN>(p, w);
            const unsigned long long deadline = g_globaltimer() + p.watchdog_ns;
            const int buf = u % NB;
            if (ok) ok = __all_sync(0xffffffffu, g_wait(&acc_full[buf], (u / NB) & 1, deadline));
            if (ok) {
                tc_fence_after();
                for (int mt = 0; mt < (x.two ? 2 : 1); ++mt) {
                    const int mrow0 = x.m0 + mt * kGemmBM + quad * 32;  // this warp's first row
                    const int rmax = min(32, p.M - mrow0);             // rows below M
                    float* part = split
                                      ? p.partials + ((static_cast<size_t>(w) * 2 + mt) * kGemmBM + quad * 32) * kGemmBN
                                      : nullptr;
                    const uint32_t tacc = tbase + lane_off + buf * L::kSetStride + mt * L::kMtStride;
#pragma unroll 1
                    for (int c = 0; c < (p.paired_I ? BN / 64 : BN / 32); ++c) {
                        // thread = row in TMEM -> a row-major 32 x 32 block in shared
                        // memory -> 4 rows of 8 float4 per warp instruction
                        float v[32];
                        tmem_ld32(tacc + c * 32, v);
                        if (p.paired_I) {
                            // gate column j and up column j + BN / 2: SiLU(gate) * up,
                            // each rounded to bf16 first as the unfused path stores them
                            float u[32];
                            tmem_ld32(tacc + BN / 2 + c * 32, u);
                            tmem_ld_wait();
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] = silu_times(bf16_round(v[i]), bf16_round(u[i]));
                        }
                        tmem_ld_wait();
#pragma unroll
                        for (int i = 0; i < 8; ++i)
                            *reinterpret_cast<float4*>(stg + lane * kGStageLd + 4 * i) =
                                make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
                        __syncwarp();
                        const int n = x.n0 + c * 32 + 4 * c4;
                        if (part) {  // rows at or past M are never read back
#pragma unroll
                            for (int q = 0; q < 8; ++q) {
                                const int rr = 4 * q + sub;
                                if (rr < rmax)
                                    *reinterpret_cast<float4*>(part + rr * kGemmBN + c * 32 + 4 * c4) =
                                        *reinterpret_cast<const float4*>(stg + rr * kGStageLd + 4 * c4);
                            }
                        } else {
                            float4 acc[8];
#pragma unroll
                            for (int q = 0; q < 8; ++q)
                                acc[q] = *reinterpret_cast<const float4*>(stg + (4 * q + sub) * kGStageLd + 4 * c4);
                            store_rows4(p, mrow0, sub, rmax, n, acc);
                        }
                        __syncwarp();
                    }
                }
            }
            tc_fence_before();
            mbar_arrive(&acc_empty[buf]);  // the MMA may refill this accumulator set
            if (split) {
                // Publish this split's partial: the barrier orders the CTA's partial
                // stores before one thread's fence and counter increment.  The launch
                // is cooperative (every unit's CTA is resident), so each split can
                // wait for its siblings; then split s adds rows
                // [s R / S, (s + 1) R / S) of the tile over every split, in split
                // order (R = rows of the pair below M).
                epi_bar();
                if (threadIdx.x == 64) {
                    __threadfence();
                    atomicAdd(p.counters + x.tile, 1);
                    bool all = false;
                    while (ok && !all) {
                        int seen;
                        asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(seen) : "l"(p.counters + x.tile) : "memory");
                        all = seen >= p.splits;
                        if (!all && g_globaltimer() > deadline) ok = false;
                    }
                    *last_flag = ok ? 1 : 0;
                }
                epi_bar();
                ok = ok && *last_flag != 0;
                if (ok) {
                    __threadfence();
                    const int R = min(2 * kGemmBM, p.M - x.m0);
                    const int r0 = x.split * R / p.splits, r1 = (x.split + 1) * R / p.splits;
                    const int n = x.n0 + 4 * lane;
                    float bias[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        bias[e] = (p.bias && n + e < p.N) ? __bfloat162float(p.bias[n + e]) : 0.f;
                    const size_t split_stride = 2 * kGemmBM * kGemmBN;
                    const float* base = p.partials + static_cast<size_t>(x.tile) * p.splits * split_stride;
                    // warps 2..5 take rows r0 + (warp - 2) + 4 i, kRG at a time
#pragma unroll 1
                    for (int rb = r0 + (warp - 2); rb < r1; rb += 4 * kRG) {
                        float4 a[kRG];
#pragma unroll
                        for (int i = 0; i < kRG; ++i) a[i] = make_float4(0.f, 0.f, 0.f, 0.f);
                        for (int sp = 0; sp < p.splits; ++sp) {  // fixed order
                            float4 f[kRG];
#pragma unroll
                            for (int i = 0; i < kRG; ++i) {
                                const int r = rb + 4 * i;
                                f[i] = r < r1 ? __ldcg(reinterpret_cast<const float4*>(
                                                    base + sp * split_stride + static_cast<size_t>(r) * kGemmBN) + lane)
                                              : make_float4(0.f, 0.f, 0.f, 0.f);
                            }
#pragma unroll
                            for (int i = 0; i < kRG; ++i) {
                                a[i].x += f[i].x;
                                a[i].y += f[i].y;
                                a[i].z += f[i].z;
                                a[i].w += f[i].w;
                            }
                        }
#pragma unroll
                        for (int i = 0; i < kRG; ++i) {
                            a[i].x += bias[0];
                            a[i].y += bias[1];
                            a[i].z += bias[2];
                            a[i].w += bias[3];
                        }
                        // pair row r = tile row (r >= 128: second tile) -> global row m0 + r
                        store_rows_strided(p, x.m0 + rb, 4, min(kRG, (r1 - rb + 3) / 4), n, a);
                    }
                }
            }
        }
        if (!ok) fail(5);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tbase, 512);
}


// ---------------------------------------------------------------- thin GEMM
// M <= 256 rows.  The roles swap: W is the A operand (128 of its rows per
// instruction) and all of X, Mp rows, the B operand (N = Mp).  A unit is one
// or two 128-row blocks of W -- two consecutive blocks, or for the gate/up
// projection a gate block and the matching up block -- over one range of K;
// the blocks share each X tile, so two blocks halve the X traffic per weight
// byte.  Each 64-wide K step loads the unit's W tiles (16 KB each) and one X
// tile of Mp x 128 B.  The `splits` units of a block (pair) are the CTAs of
// one thread-block cluster: after the main loop each stages its fp32
// accumulators in its own shared memory (the stage ring is idle by then; the
// staging area may reach past it), and after a cluster barrier CTA r adds
// rows [r M / S, (r + 1) M / S) over the S CTAs' copies in rank order,
// applies the epilogue and writes bf16.  No partial sum leaves the cluster
// and the result does not depend on timing.
constexpr int kTTileW = 128 * kGemmBK * 2;  // 16 KB: 128 rows of W x 64 K
constexpr int kTMaxStages = 8;
constexpr int kTBarBytes = 256;             // barriers, TMEM slot, abort flag
constexpr int kTSmemMax = 232448;
constexpr int kTRegionMax = kTSmemMax - 1024 - kTBarBytes;  // ring / staging area
// Every plan uses more than half of an SM's shared memory, so each SM holds
// one CTA and no CTA waits on another cluster's for TMEM.
static_assert(kTMaxStages * (kTTileW + 16 * kGemmBK * 2) > 233472 / 2, "one CTA per SM");

__host__ __device__ constexpr int thin_stage_bytes(int Mp, int wblocks)
{
    return wblocks * kTTileW + Mp * kGemmBK * 2;
}

__host__ __device__ constexpr size_t thin_staging_bytes(int M, int wblocks)
{
    return static_cast<size_t>(wblocks) * M * 128 * 4;
}

__device__ __forceinline__ void add4(float4& a, const float4& b)
{
    a.x += b.x;
    a.y += b.y;
    a.z += b.z;
    a.w += b.w;
}

// four consecutive staged values of row t, summed over the cluster's S CTAs
// in rank order (stage: fp32 [rows][128] at shared address `base` in every
// CTA).  All S loads are issued before the first addition.
template <int S>
__device__ __forceinline__ float4 cluster_sum4(uint32_t base, int t, int col)
{
    const uint32_t a = base + static_cast<uint32_t>(t * 128 + col) * 4u;
    float4 v[S];
#pragma unroll
    for (int r = 0; r < S; ++r) v[r] = ld_dsmem_f4(dsmem_addr(a, r));
#pragma unroll
    for (int r = 1; r < S; ++r) add4(v[0], v[r]);
    return v[0];
}

__device__ __forceinline__ void store_bf16x4(__nv_bfloat16* dst, float a, float b, float c, float d)
{
    *reinterpret_cast<uint2*>(dst) = make_uint2(pack_bf16x2(a, b), pack_bf16x2(c, d));
}

// Residual epilogue of one staged block: out[t][wb + j] += sum, rows
// [t0, t1), 4 columns per thread (e = 0..127: column group e mod 32, row
// phase e / 32).  Rows go in batches whose loads (about 8 in flight per thread)
// are all issued before the first use.
template <int S>
__device__ __forceinline__ void epi_residual(const ThinParams& p, uint32_t sbase, int wb, int nv, int t0,
                                             int t1, int e)
{
    constexpr int kB = 8 / S > 0 ? 8 / S : 1;
    const int j4 = 4 * (e & 31);
    if (j4 >= nv) return;
    for (int tb = t0 + (e >> 5); tb < t1; tb += 4 * kB) {
        uint2 old[kB];
        float4 a[kB];
#pragma unroll
        for (int b = 0; b < kB; ++b)
            if (tb + 4 * b < t1)
                old[b] = *reinterpret_cast<const uint2*>(p.out + static_cast<size_t>(tb + 4 * b) * p.Nw + wb + j4);
#pragma unroll
        for (int b = 0; b < kB; ++b)
            if (tb + 4 * b < t1) a[b] = cluster_sum4<S>(sbase, tb + 4 * b, j4);
#pragma unroll
        for (int b = 0; b < kB; ++b)
            if (tb + 4 * b < t1) {
                const float2 lo = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&old[b].x));
                const float2 hi = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&old[b].y));
                store_bf16x4(p.out + static_cast<size_t>(tb + 4 * b) * p.Nw + wb + j4, lo.x + a[b].x,
                             lo.y + a[b].y, hi.x + a[b].z, hi.y + a[b].w);
            }
    }
}

// QKV epilogue of one staged block (W rows wb.., whole heads): bias added and
// rounded to bf16 where the projection would be stored, q and k heads
// rotated by the rows' (cos, sin) table, written to q / k / v in [M][H][d].
// 16 threads per row: thread g takes pairs (k, k + d/2), k = 4 (g mod d/8)
// .. +3, of the block's head g / (d/8).
template <int S>
__device__ __forceinline__ void epi_qkv(const ThinParams& p, uint32_t sbase, int wb, int t0, int t1, int e)
{
    constexpr int kB = 8 / S > 0 ? 8 / S : 1;
    const int half = p.d / 2, gph = half / 4;  // 4-pair groups per head
    const int g = e & 15, lh = g / gph, k = 4 * (g - lh * gph);
    const int c1 = lh * p.d + k, f1 = wb + c1;  // block column, W row of the first value
    if (f1 >= p.Nw) return;
    const int head = f1 / p.d;
    const bool rotate = head < p.Hq + p.Hkv;
    __nv_bfloat16* dst0 = head < p.Hq ? p.q + static_cast<size_t>(head) * p.d
                        : rotate      ? p.k + static_cast<size_t>(head - p.Hq) * p.d
                                      : p.v + static_cast<size_t>(head - p.Hq - p.Hkv) * p.d;
    const int row_stride = (head < p.Hq ? p.Hq : p.Hkv) * p.d;
    float b1[4], b2[4];  // this thread's bias values, the same for every row
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        b1[i] = p.bias ? __bfloat162float(p.bias[f1 + i]) : 0.f;
        b2[i] = p.bias ? __bfloat162float(p.bias[f1 + half + i]) : 0.f;
    }
    for (int tb = t0 + (e >> 4); tb < t1; tb += 8 * kB) {
        float4 a1[kB], a2[kB], cs[kB][2];
#pragma unroll
        for (int b = 0; b < kB; ++b) {
            const int t = tb + 8 * b;
            if (t < t1 && rotate) {
                const float4* r4 = reinterpret_cast<const float4*>(p.rope + static_cast<size_t>(t) * half + k);
                cs[b][0] = r4[0];  // (cos, sin) of pairs k, k + 1
                cs[b][1] = r4[1];  // of pairs k + 2, k + 3
            }
        }
#pragma unroll
        for (int b = 0; b < kB; ++b) {
            const int t = tb + 8 * b;
            if (t < t1) {
                a1[b] = cluster_sum4<S>(sbase, t, c1);
                a2[b] = cluster_sum4<S>(sbase, t, c1 + half);
            }
        }
#pragma unroll
        for (int b = 0; b < kB; ++b) {
            const int t = tb + 8 * b;
            if (t >= t1) continue;
            float x1[4] = {a1[b].x, a1[b].y, a1[b].z, a1[b].w}, x2[4] = {a2[b].x, a2[b].y, a2[b].z, a2[b].w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                x1[i] = bf16_round(x1[i] + b1[i]);
                x2[i] = bf16_round(x2[i] + b2[i]);
            }
            if (rotate) {
                const float c[4] = {cs[b][0].x, cs[b][0].z, cs[b][1].x, cs[b][1].z};
                const float sn[4] = {cs[b][0].y, cs[b][0].w, cs[b][1].y, cs[b][1].w};
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float o1 = x1[i] * c[i] - x2[i] * sn[i];
                    const float o2 = x2[i] * c[i] + x1[i] * sn[i];
                    x1[i] = o1;
                    x2[i] = o2;
                }
            }
            __nv_bfloat16* dst = dst0 + static_cast<size_t>(t) * row_stride;
            store_bf16x4(dst + k, x1[0], x1[1], x1[2], x1[3]);
            store_bf16x4(dst + k + half, x2[0], x2[1], x2[2], x2[3]);
        }
    }
}

// SiLU * up from the staged gate (sbase) and up (ubase) blocks, summed over
// the cluster: out[t][col0 + j] for j < nv (layout as epi_residual's).
template <int S>
__device__ __forceinline__ void epi_silu(const ThinParams& p, uint32_t sbase, uint32_t ubase, int col0, int nv,
                                         int t0, int t1, int e)
{
    constexpr int kB = 8 / S > 0 ? 8 / S : 1;
    const int j4 = 4 * (e & 31);
    if (j4 >= nv) return;
    for (int tb = t0 + (e >> 5); tb < t1; tb += 4 * kB) {
        float4 g[kB], u[kB];
#pragma unroll
        for (int b = 0; b < kB; ++b)
            if (tb + 4 * b < t1) {
                g[b] = cluster_sum4<S>(sbase, tb + 4 * b, j4);
                u[b] = cluster_sum4<S>(ubase, tb + 4 * b, j4);
            }
#pragma unroll
        for (int b = 0; b < kB; ++b)
            if (tb + 4 * b < t1)
                store_bf16x4(p.out + static_cast<size_t>(tb + 4 * b) * p.paired_I + col0 + j4,
                             silu_times(bf16_round(g[b].x), bf16_round(u[b].x)),
                             silu_times(bf16_round(g[b].y), bf16_round(u[b].y)),
                             silu_times(bf16_round(g[b].z), bf16_round(u[b].z)),
                             silu_times(bf16_round(g[b].w), bf16_round(u[b].w)));
    }
}

// Part 2 of the epilogue for a cluster of S CTAs (S in {1, 2, 4, 8}).
template <int S>
__device__ __forceinline__ void epi_part2(const ThinParams& p, uint32_t base, uint32_t blk, int nacc, int wb0,
                                          int wb1, int nv0, int nv1, int t0, int t1, int e)
{
    if (p.op == kThinSilu) {
        epi_silu<S>(p, base, base + blk, wb0, nv0, t0, t1, e);
        return;
    }
    for (int a = 0; a < nacc; ++a) {
        if (p.op == kThinResidual) epi_residual<S>(p, base + a * blk, a ? wb1 : wb0, a ? nv1 : nv0, t0, t1, e);
        else epi_qkv<S>(p, base + a * blk, a ? wb1 : wb0, t0, t1, e);
    }
}

__global__ void __launch_bounds__(kGThreads, 1)
    gemm_thin_tc(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_w,
                 const ThinParams p)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
    const bool paired = p.paired_I > 0;
    const int S = p.stages;
    const int stage_bytes = thin_stage_bytes(p.Mp, p.wblocks);
    const int x_off = p.wblocks * kTTileW;  // the X tile's offset in a stage
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + p.region);
    uint64_t* full = bars;            // stage loaded
    uint64_t* empty = bars + S;       // stage read by its MMAs
    uint64_t* acc_full = bars + 2 * S;
    uint64_t* drain = acc_full + 1;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int tile = blockIdx.x / p.splits, split = blockIdx.x - tile * p.splits;  // split = cluster rank
    const int ks0 = split * p.kps, ks1 = min(p.k_steps, ks0 + p.kps);
    // the unit's W row blocks and how many of their rows are outputs
    int wb0, wb1, nv0, nv1;
    if (paired) {
        wb0 = 128 * tile;
        wb1 = p.paired_I + wb0;
        nv0 = nv1 = min(128, p.paired_I - wb0);
    } else {
        wb0 = 128 * p.wblocks * tile;
        wb1 = wb0 + 128;
        nv0 = min(128, p.Nw - wb0);
        nv1 = p.wblocks == 2 ? max(0, min(128, p.Nw - wb1)) : 0;
    }
    const int nacc = nv1 > 0 ? 2 : 1;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int i = 0; i < S; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        mbar_init(acc_full, 1);
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, 512);
        tmem_relinquish();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tmem_slot;
    const unsigned long long deadline = g_globaltimer() + p.watchdog_ns;
    auto fail = [&](int site) {
        if (atomicExch(const_cast<int*>(abort_flag), 1) == 0)
            *reinterpret_cast<volatile int32_t*>(p.status) = DEV_TIMEOUT_GEMM | (site << 8);
    };
    // the next kernel may start launching (it waits for this one's completion
    // before touching what this one writes)
    pdl_launch_dependents();

    bool ok = true;
    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            tma_prefetch_desc(&tm_x);
            tma_prefetch_desc(&tm_w);
            const uint32_t tx = nacc * kTTileW + p.Mp * kGemmBK * 2;
            // The weights do not depend on the previous kernel of the stream:
            // the first ring's worth of W tiles is requested before waiting
            // for it (a no-op unless launched programmatically), X after.
            const int pre = min(S, ks1 - ks0);
            for (int n = 0; n < pre; ++n) {
                uint8_t* base = sm + n * stage_bytes;
                mbar_arrive_expect_tx(&full[n], tx);
                const int kc = (ks0 + n) * kGemmBK;
                tma_load_4d(base, &tm_w, &full[n], kc, wb0, 0, 0);
                if (nacc == 2) tma_load_4d(base + kTTileW, &tm_w, &full[n], kc, wb1, 0, 0);
            }
            pdl_wait();
            for (int n = 0; n < pre; ++n)
                tma_load_4d(sm + n * stage_bytes + x_off, &tm_x, &full[n], (ks0 + n) * kGemmBK, 0, 0, 0);
            int n = pre;
            for (int ks = ks0 + pre; ks < ks1; ++ks, ++n) {
                if (*abort_flag) break;
                const int s = n % S, use = n / S;
                if (use >= 1 && !g_wait(&empty[s], (use - 1) & 1, deadline)) {
                    fail(6);
                    break;
                }
                uint8_t* base = sm + s * stage_bytes;
                mbar_arrive_expect_tx(&full[s], tx);
                const int kc = ks * kGemmBK;
                tma_load_4d(base, &tm_w, &full[s], kc, wb0, 0, 0);
                if (nacc == 2) tma_load_4d(base + kTTileW, &tm_w, &full[s], kc, wb1, 0, 0);
                tma_load_4d(base + x_off, &tm_x, &full[s], kc, 0, 0, 0);
            }
            // let every copy land before the stages are reused or the CTA's
            // memory goes away: the last use of stage s is the largest one issued
            const unsigned long long dl = g_globaltimer() + p.watchdog_ns;
            for (int s = 0; s < S && s < n; ++s) g_wait(&full[s], ((n - 1 - s) / S) & 1, dl);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t id = idesc_bf16_f32(128, p.Mp, false, false);
            const uint32_t s0 = smem_addr(sm);
            int n = 0;
            for (int ks = ks0; ks < ks1; ++ks, ++n) {
                const int s = n % S;
                if (!(ok = g_wait(&full[s], (n / S) & 1, deadline))) break;
                tc_fence_after();
                const uint32_t sa = s0 + s * stage_bytes;
                const uint64_t da0 = sdesc_sw128(sa, 16, 1024);
                const uint64_t da1 = sdesc_sw128(sa + kTTileW, 16, 1024);
                const uint64_t dx = sdesc_sw128(sa + x_off, 16, 1024);
#pragma unroll
                for (int kk = 0; kk < kGemmBK / 16; ++kk) {
                    const uint32_t acc = (ks > ks0 || kk > 0) ? 1u : 0u;
                    umma_bf16(tbase, da0 + 2 * kk, dx + 2 * kk, id, acc);
                    if (nacc == 2) umma_bf16(tbase + 256, da1 + 2 * kk, dx + 2 * kk, id, acc);
                }
                umma_commit(&empty[s]);
            }
            if (ok) umma_commit(acc_full);
            else fail(7);
            umma_commit(drain);
            g_wait(drain, 0, g_globaltimer() + p.watchdog_ns);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue (warps 2..5), part 1
        // thread = W row (TMEM lane); each 32-column TMEM load holds 32 rows of X
        const int quad = warp & 3;
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        const int r = quad * 32 + lane;
        const int chunks = (p.M + 31) / 32;
        ok = __all_sync(0xffffffffu, g_wait(acc_full, 0, deadline));
        if (!ok) fail(8);
        if (ok) tc_fence_after();
        if (ok && p.op == kThinSilu && p.splits == 1) {
            // the whole K range is here: SiLU(gate) * up straight from TMEM,
            // staged as bf16 rows, then written out with 16-byte stores, 16
            // threads per row
            __nv_bfloat16* stage = reinterpret_cast<__nv_bfloat16*>(sm);  // [M][128]
#pragma unroll 1
            for (int c = 0; c < chunks; ++c) {
                float g[32], u[32];
                tmem_ld32(tbase + lane_off + 32 * c, g);
                tmem_ld32(tbase + lane_off + 256 + 32 * c, u);
                tmem_ld_wait();
                // the 32 values first (independent chains the compiler can
                // interleave), then the predicated stores
#pragma unroll
                for (int j = 0; j < 32; ++j) g[j] = silu_times(bf16_round(g[j]), bf16_round(u[j]));
                uint16_t* srow = reinterpret_cast<uint16_t*>(stage) + (32 * c) * 128 + r;
                if (32 * c + 32 <= p.M) {
#pragma unroll
                    for (int j = 0; j < 32; ++j) srow[j * 128] = static_cast<uint16_t>(bf16_rne_bits(g[j]));
                } else {
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (32 * c + j < p.M) srow[j * 128] = static_cast<uint16_t>(bf16_rne_bits(g[j]));
                }
            }
            epi_bar();
            const int e = threadIdx.x - 64, c16 = e & 15;
            if (8 * c16 < nv0)
                for (int t = e >> 4; t < p.M; t += 8)
                    *reinterpret_cast<uint4*>(p.out + static_cast<size_t>(t) * p.paired_I + wb0 + 8 * c16) =
                        *reinterpret_cast<const uint4*>(stage + t * 128 + 8 * c16);
        } else if (ok) {
            float* stage = reinterpret_cast<float*>(sm);  // [nacc][M][128]
            for (int a = 0; a < nacc; ++a)
#pragma unroll 1
                for (int c = 0; c < chunks; ++c) {
                    float v[32];
                    tmem_ld32(tbase + lane_off + 256 * a + 32 * c, v);
                    tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int t = 32 * c + j;
                        if (t < p.M) stage[(a * p.M + t) * 128 + r] = v[j];
                    }
                }
        }
    }
    // every CTA of the cluster has staged its accumulators
    cluster_sync();
    if (warp >= 2 && !(p.op == kThinSilu && p.splits == 1)) {
        // ------------------------------------------------------------ epilogue, part 2
        // this CTA's share of the rows, summed over the cluster in rank order
        const int e = threadIdx.x - 64;  // 0..127
        const int t0 = split * p.M / p.splits, t1 = (split + 1) * p.M / p.splits;
        const uint32_t base = smem_addr(sm), blk = static_cast<uint32_t>(p.M) * 128u * 4u;
        switch (p.splits) {
            case 1: epi_part2<1>(p, base, blk, nacc, wb0, wb1, nv0, nv1, t0, t1, e); break;
            case 2: epi_part2<2>(p, base, blk, nacc, wb0, wb1, nv0, nv1, t0, t1, e); break;
            case 4: epi_part2<4>(p, base, blk, nacc, wb0, wb1, nv0, nv1, t0, t1, e); break;
            default: epi_part2<8>(p, base, blk, nacc, wb0, wb1, nv0, nv1, t0, t1, e); break;
        }
    }
    // no CTA leaves while the others may still read its shared memory
    cluster_sync();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tbase, 512);
}

}  // namespace

GemmPlan gemm_plan(int M, int N, int K, int sms)
{
    GemmPlan g{};
    g.m_pairs = (M + 2 * kGemmBM - 1) / (2 * kGemmBM);
    g.k_steps = (K + kGemmBK - 1) / kGemmBK;
    // Wider tiles (192 or 256 W rows) when the 128-wide ones take several
    // rounds on the SMs and fewer rounds of wider ones cost less: a 256-wide
    // unit measured 1.82x a 128-wide one (twice the work), a 192-wide one
    // 1.41x.  Only with K long enough to hide the epilogue they cannot overlap
    // (one accumulator set) and 128-byte aligned rows (at K = 200, or with
    // K = 3592, they were slower).
    g.bn = kGemmBN;
    const int narrow = (N + kGemmBN - 1) / kGemmBN * g.m_pairs;
    if (narrow >= sms && g.k_steps >= 32 && (K % 64) == 0) {
        double best = (narrow + sms - 1) / sms;
        const int widths[2] = {192, 256};
        const double unit_cost[2] = {1.41, 1.82};
        for (int i = 0; i < 2; ++i) {
            const int t = (N + widths[i] - 1) / widths[i] * g.m_pairs;
            const double cost = ((t + sms - 1) / sms) * unit_cost[i];
            if (cost < best - 0.05) {
                best = cost;
                g.bn = widths[i];
            }
        }
    }
    g.n_tiles = (N + g.bn - 1) / g.bn;
    const int tiles = g.n_tiles * g.m_pairs;
    // split K only while the tiles alone leave SMs idle, into as many ranges as
    // keep every unit in one wave
    int splits = tiles >= sms ? 1 : sms / tiles;
    splits = splits < 1 ? 1 : (splits > g.k_steps ? g.k_steps : splits);
    g.kps = (g.k_steps + splits - 1) / splits;
    g.splits = (g.k_steps + g.kps - 1) / g.kps;
    g.units = tiles * g.splits;
    g.partial_bytes = g.splits > 1 ? static_cast<size_t>(g.units) * 2 * kGemmBM * kGemmBN * 4 : 0;
    g.counters = g.splits > 1 ? tiles : 0;
    return g;
}

cudaError_t gemm_prepare()
{
    cudaError_t e = cudaFuncSetAttribute(gemm_bf16_tc<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         GLayout<128>::kAlloc);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(gemm_bf16_tc<192>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 GLayout<192>::kAlloc);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(gemm_bf16_tc<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                GLayout<256>::kAlloc);
}

cudaError_t launch_gemm(const CUtensorMap& tm_x, const CUtensorMap& tm_w, const GemmParams& p,
                        int sms, cudaStream_t st)
{
    if (p.units <= 0) return cudaSuccess;
    if (p.bn != 128 && p.bn != 192 && p.bn != 256) return cudaErrorInvalidValue;
    if (p.paired_I && (p.splits != 1 || p.paired_I != p.N || p.bias || p.add)) return cudaErrorInvalidValue;
    const int grid = p.units < sms ? p.units : sms;
    if (p.bn != 128) {
        if (p.splits != 1) return cudaErrorInvalidValue;
        if (p.bn == 192)
            gemm_bf16_tc<192><<<grid, kGThreads, GLayout<192>::kAlloc, st>>>(tm_x, tm_w, p);
        else
            gemm_bf16_tc<256><<<grid, kGThreads, GLayout<256>::kAlloc, st>>>(tm_x, tm_w, p);
        return cudaGetLastError();
    }
    if (p.splits == 1) {
        gemm_bf16_tc<128><<<grid, kGThreads, GLayout<128>::kAlloc, st>>>(tm_x, tm_w, p);
        return cudaGetLastError();
    }
    // split K: the splits of a tile wait for one another, so every unit's CTA
    // must be resident at once (units <= SMs, one CTA per SM)
    if (p.units > sms) return cudaErrorInvalidConfiguration;
    CUtensorMap a = tm_x, b = tm_w;
    GemmParams q = p;
    void* args[] = {&a, &b, &q};
    return cudaLaunchCooperativeKernel(reinterpret_cast<const void*>(gemm_bf16_tc<128>), dim3(grid),
                                       dim3(kGThreads), args, GLayout<128>::kAlloc, st);
}

namespace {

// clusters of each size (1..kThinMaxSplits CTAs) that one device holds at
// once with the thin kernel's shared memory, measured at set-up per device
constexpr int kThinMaxDevices = 64;
int g_thin_clusters[kThinMaxDevices][kThinMaxSplits + 1] = {};

int thin_max_clusters(int size, int sms)
{
    int dev = 0;
    if (cudaGetDevice(&dev) == cudaSuccess && dev >= 0 && dev < kThinMaxDevices && g_thin_clusters[dev][size] > 0)
        return g_thin_clusters[dev][size];
    return sms / size / 2;  // not measured: assume half the SMs usable
}

}  // namespace

ThinPlan thin_plan(int M, int Nw, int K, int sms, int paired_I)
{
    // The unit shape (one or two W blocks) and the split count (the cluster
    // size) are chosen by a streaming model fitted to measured launches: the
    // time is a fixed cost per launch plus the bytes the CTAs load -- every
    // weight byte once, the X tile once per CTA and K step -- at
    // min(CTAs x 65 GB/s, 7.3 TB/s), with a wave per max-active-cluster
    // count of clusters.
    const bool paired = paired_I > 0;
    const int Mp = (M + 15) / 16 * 16;
    const int k_steps = (K + kGemmBK - 1) / kGemmBK;
    const double w_bytes = 2.0 * K * (paired ? 2.0 * paired_I : static_cast<double>(Nw));
    ThinPlan best{};
    double best_us = 1e30;
    for (int wb = paired ? 2 : 1; wb <= 2; ++wb) {
        const int tiles = paired ? (paired_I + 127) / 128 : (Nw + 128 * wb - 1) / (128 * wb);
        const int sb = thin_stage_bytes(Mp, wb);
        const int stages = std::min(kTMaxStages, kTRegionMax / sb);
        if (stages < 2) continue;
        for (int s = 1; s <= kThinMaxSplits; s *= 2) {
            const int kps = (k_steps + s - 1) / s;
            if ((s - 1) * kps >= k_steps) continue;  // every split gets K steps
            const bool staged = !(paired && s == 1);
            if (staged && thin_staging_bytes(M, wb) > static_cast<size_t>(kTRegionMax)) continue;
            const int ctas = tiles * s;
            const int per_wave = std::max(1, thin_max_clusters(s, sms));
            const int waves = (tiles + per_wave - 1) / per_wave;
            const int active = std::min(tiles, per_wave) * s;
            const double bytes = w_bytes + static_cast<double>(ctas) * Mp * kps * kGemmBK * 2;
            const double rate = std::min(active * 65e3, 7.3e6);  // bytes per us
            const double us = 4.0 * waves + (s > 1 ? 1.0 : 0.0) + bytes / rate;
            if (us < best_us - 0.05) {
                best_us = us;
                best.tiles = tiles;
                best.k_steps = k_steps;
                best.kps = kps;
                best.splits = s;
                best.Mp = Mp;
                best.stages = stages;
                best.wblocks = wb;
                const size_t ring = static_cast<size_t>(stages) * sb;
                best.region = std::max(ring, staged ? thin_staging_bytes(M, wb) : 0);
                best.region = (best.region + 1023) / 1024 * 1024;
                best.smem = best.region + kTBarBytes + 1024;
            }
        }
    }
    return best;
}

cudaError_t thin_prepare()
{
    cudaError_t e = cudaFuncSetAttribute(gemm_thin_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, kTSmemMax);
    if (e != cudaSuccess) return e;
    int dev = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if (dev < 0 || dev >= kThinMaxDevices) return cudaSuccess;  // plans fall back to a guess
    for (int s = 1; s <= kThinMaxSplits; ++s) {
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3(s);
        cfg.blockDim = dim3(kGThreads);
        cfg.dynamicSmemBytes = kTSmemMax;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = s;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int n = 0;
        if ((e = cudaOccupancyMaxActiveClusters(&n, gemm_thin_tc, &cfg)) != cudaSuccess) return e;
        g_thin_clusters[dev][s] = n;
    }
    return cudaSuccess;
}

cudaError_t launch_thin_gemm(const CUtensorMap& tm_x, const CUtensorMap& tm_w, const ThinParams& p,
                             size_t smem, cudaStream_t st)
{
    const bool paired = p.paired_I > 0;
    if (p.wblocks != 1 && p.wblocks != 2) return cudaErrorInvalidValue;
    const int tiles = paired ? (p.paired_I + 127) / 128 : (p.Nw + 128 * p.wblocks - 1) / (128 * p.wblocks);
    if (tiles <= 0) return cudaSuccess;
    const size_t ring = static_cast<size_t>(p.stages) * thin_stage_bytes(p.Mp, p.wblocks);
    const bool staged = !(p.op == kThinSilu && p.splits == 1);
    if (p.M < 1 || p.M > kThinMaxRows || p.Mp != (p.M + 15) / 16 * 16 || p.stages < 2 ||
        p.stages > kTMaxStages || (p.splits != 1 && p.splits != 2 && p.splits != 4 && p.splits != 8) ||
        (p.splits - 1) * p.kps >= p.k_steps || p.splits * p.kps < p.k_steps ||
        (!p.out && p.op != kThinQkvRope) || (p.op == kThinSilu) != paired || (paired && p.wblocks != 2) ||
        (paired && (p.paired_I & 7) != 0) || (!paired && (p.Nw & 3) != 0) ||
        (p.op == kThinQkvRope && (!p.q || !p.k || !p.v || !p.rope || (p.d != 64 && p.d != 128) ||
                                  p.Nw != (p.Hq + 2 * p.Hkv) * p.d)) ||
        ring > p.region || (staged && thin_staging_bytes(p.M, p.wblocks) > p.region) || p.region % 1024 != 0 ||
        p.region + kTBarBytes + 1024 > smem || smem > static_cast<size_t>(kTSmemMax))
        return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(tiles * p.splits);
    cfg.blockDim = dim3(kGThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = p.splits;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, gemm_thin_tc, tm_x, tm_w, p);
}

}  // namespace statekv
