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
//     split into ranges: every split writes an fp32 partial of its tile, and
//     the last split to finish (an atomic counter per tile, no waiting) adds
//     the partials in split order, so the result does not depend on timing;
//   - one CTA per SM walks the units; TMEM holds two accumulator sets, so the
//     epilogue of one unit overlaps the main loop of the next.
// 192 threads: warp 0 issues the TMA loads (a four-stage ring of 48 KB: X rows
// m0..m0+127, X rows m0+128..m0+255, W rows n0..n0+127, 64 K-columns each,
// 128-byte swizzle), warp 1 allocates TMEM and issues tcgen05.mma
// (128 x 128 x 16, both operands K-major in shared memory), warps 2..5 read
// the accumulators (one TMEM lane quadrant each, thread = row) and write D or
// the fp32 partials.  Every mbarrier wait is bounded by the watchdog; on
// expiry the CTA records DEV_TIMEOUT_GEMM, drains and exits.
#include "sm103_ptx.cuh"
#include "statekv_kernels.cuh"

namespace statekv {
namespace {

using namespace ptx;

constexpr int kGThreads = 192;
constexpr int kGStages = 4;
constexpr int kGTileA = kGemmBM * kGemmBK * 2;        // 16 KB: 128 rows of X x 64 K
constexpr int kGTileB = kGemmBN * kGemmBK * 2;        // 16 KB: 128 rows of W x 64 K
constexpr int kGStageBytes = 2 * kGTileA + kGTileB;   // 48 KB
// epilogue staging: per epilogue warp a 32 x 36 fp32 block (row-major, 16-byte
// rows padded by one float4 against bank conflicts) turns thread-per-row TMEM
// reads into row-contiguous global stores
constexpr int kGStageLd = 36;
constexpr int kRG = 8;  // rows per group of the split-K reduction (2 kRG loads in flight)
constexpr int kGOffEpi = kGStages * kGStageBytes;
constexpr int kGOffBar = kGOffEpi + 4 * 32 * kGStageLd * 4;
constexpr int kGNumBars = 2 * kGStages + 5;           // full[4] empty[4] acc_full[2] acc_empty[2] drain
constexpr int kGOffMisc = kGOffBar + kGNumBars * 8;
constexpr int kGBytes = kGOffMisc + 16;
constexpr int kGAlloc = kGBytes + 1024;               // room to align the base to 1 KB
static_assert(kGAlloc <= 232448, "shared memory budget");
static_assert(kGStageBytes % 1024 == 0 && kGTileA % 1024 == 0, "swizzle atoms stay aligned");

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

__device__ __forceinline__ GemmUnit gemm_unit(const GemmParams& p, int w)
{
    GemmUnit x;
    x.tile = w / p.splits;
    x.split = w - x.tile * p.splits;
    x.n0 = (x.tile % p.n_tiles) * kGemmBN;
    x.m0 = (x.tile / p.n_tiles) * 2 * kGemmBM;
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

__global__ void __launch_bounds__(kGThreads, 1)
    gemm_bf16_tc(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_w,
                 const GemmParams p)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + kGOffBar);
    uint64_t* full = bars;                     // stage loaded
    uint64_t* empty = bars + kGStages;         // stage read by its MMAs
    uint64_t* acc_full = bars + 2 * kGStages;  // accumulator set complete
    uint64_t* acc_empty = acc_full + 2;        // accumulator set read out
    uint64_t* drain = acc_full + 4;            // every MMA of the CTA has completed
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + kGOffMisc);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(sm + kGOffMisc + 4);
    volatile int* last_flag = reinterpret_cast<volatile int*>(sm + kGOffMisc + 8);

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
                const GemmUnit x = gemm_unit(p, w);
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
                    tma_load_4d(base + 2 * kGTileA, &tm_w, &full[s], kc, x.n0, 0, 0);
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
            constexpr uint32_t kId = idesc_bf16_f32(kGemmBM, kGemmBN, false, false);
            const uint32_t s0 = smem_addr(sm);
            bool ok = true;
            int n = 0, u = 0, site = 3;
            for (int w = blockIdx.x; ok && w < p.units; w += gridDim.x, ++u) {
                const GemmUnit x = gemm_unit(p, w);
                const unsigned long long deadline = g_globaltimer() + p.watchdog_ns;
                const int buf = u & 1;
                site = 4;
                if (u >= 2 && !(ok = g_wait(&acc_empty[buf], ((u - 2) >> 1) & 1, deadline))) break;
                tc_fence_after();
                const uint32_t acc0 = tbase + buf * 256, acc1 = acc0 + 128;
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
        float* stg = reinterpret_cast<float*>(sm + kGOffEpi) + (warp - 2) * 32 * kGStageLd;
        const int sub = lane >> 3, c4 = lane & 7;  // staging read-out: 4 rows x 8 float4 per instruction
        bool ok = true;
        int u = 0;
        for (int w = blockIdx.x; w < p.units; w += gridDim.x, ++u) {
            const GemmUnit x = gemm_unit(p, w);
            const unsigned long long deadline = g_globaltimer() + p.watchdog_ns;
            const int buf = u & 1;
            if (ok) ok = __all_sync(0xffffffffu, g_wait(&acc_full[buf], (u >> 1) & 1, deadline));
            if (ok) {
                tc_fence_after();
                for (int mt = 0; mt < (x.two ? 2 : 1); ++mt) {
                    const int mrow0 = x.m0 + mt * kGemmBM + quad * 32;  // this warp's first row
                    const int rmax = min(32, p.M - mrow0);             // rows below M
                    float* part = p.splits > 1
                                      ? p.partials + ((static_cast<size_t>(w) * 2 + mt) * kGemmBM + quad * 32) * kGemmBN
                                      : nullptr;
#pragma unroll 1
                    for (int c = 0; c < kGemmBN / 32; ++c) {
                        // thread = row in TMEM -> a row-major 32 x 32 block in shared
                        // memory -> 4 rows of 8 float4 per warp instruction
                        float v[32];
                        tmem_ld32(tbase + lane_off + buf * 256 + mt * 128 + c * 32, v);
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
            if (p.splits > 1) {
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
// instruction, two row blocks per unit) and the whole of X, Mp rows, the B
// operand (N = Mp), so each 64-wide K step loads two 16 KB W tiles and one
// X tile of Mp x 128 B, and both accumulators (TMEM columns [0, Mp) and
// [256, 256 + Mp)) share the X tile.  One unit per CTA: nothing waits on
// another CTA.
constexpr int kTTileW = 128 * kGemmBK * 2;  // 16 KB: 128 rows of W x 64 K
constexpr int kTMaxStages = 8;
constexpr int kTBarBytes = 256;             // barriers, TMEM slot, abort flag
constexpr int kTSmemMax = 232448;

__host__ __device__ constexpr int thin_stage_bytes(int Mp) { return 2 * kTTileW + Mp * kGemmBK * 2; }

__device__ __forceinline__ float silu_times(float g, float u) { return g / (1.f + expf(-g)) * u; }

__global__ void __launch_bounds__(kGThreads, 1)
    gemm_thin_tc(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_w,
                 const ThinParams p)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
    const int S = p.stages;
    const int stage_bytes = thin_stage_bytes(p.Mp);
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + S * stage_bytes);
    uint64_t* full = bars;            // stage loaded
    uint64_t* empty = bars + S;       // stage read by its MMAs
    uint64_t* acc_full = bars + 2 * S;
    uint64_t* drain = acc_full + 1;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int tile = blockIdx.x / p.splits, split = blockIdx.x - tile * p.splits;
    const int ks0 = split * p.kps, ks1 = min(p.k_steps, ks0 + p.kps);
    // W row blocks of the unit and the rows of each that are outputs
    int wb0, wb1, nv0, nv1;
    if (p.paired_I > 0) {
        wb0 = 128 * tile;
        wb1 = p.paired_I + 128 * tile;
        nv0 = nv1 = min(128, p.paired_I - 128 * tile);
    } else {
        wb0 = 256 * tile;
        wb1 = wb0 + 128;
        nv0 = min(128, p.Nw - wb0);
        nv1 = max(0, min(128, p.Nw - wb1));
    }
    const bool two = nv1 > 0;

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

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            tma_prefetch_desc(&tm_x);
            tma_prefetch_desc(&tm_w);
            const uint32_t tx = (two ? 2 : 1) * kTTileW + p.Mp * kGemmBK * 2;
            // The weights do not depend on the previous kernel of the stream:
            // the first ring's worth of W tiles is requested before waiting
            // for it (a no-op unless launched programmatically), X after.
            const int pre = min(S, ks1 - ks0);
            for (int n = 0; n < pre; ++n) {
                uint8_t* base = sm + n * stage_bytes;
                mbar_arrive_expect_tx(&full[n], tx);
                const int kc = (ks0 + n) * kGemmBK;
                tma_load_4d(base, &tm_w, &full[n], kc, wb0, 0, 0);
                if (two) tma_load_4d(base + kTTileW, &tm_w, &full[n], kc, wb1, 0, 0);
            }
            pdl_wait();
            for (int n = 0; n < pre; ++n)
                tma_load_4d(sm + n * stage_bytes + 2 * kTTileW, &tm_x, &full[n], (ks0 + n) * kGemmBK, 0, 0, 0);
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
                if (two) tma_load_4d(base + kTTileW, &tm_w, &full[s], kc, wb1, 0, 0);
                tma_load_4d(base + 2 * kTTileW, &tm_x, &full[s], kc, 0, 0, 0);
            }
            // let every copy land before the CTA's memory goes away: the last
            // use of stage s is the largest use issued for it
            const unsigned long long dl = g_globaltimer() + p.watchdog_ns;
            for (int s = 0; s < S && s < n; ++s) g_wait(&full[s], ((n - 1 - s) / S) & 1, dl);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t id = idesc_bf16_f32(128, p.Mp, false, false);
            const uint32_t s0 = smem_addr(sm);
            bool ok = true;
            int n = 0;
            for (int ks = ks0; ks < ks1; ++ks, ++n) {
                const int s = n % S;
                if (!(ok = g_wait(&full[s], (n / S) & 1, deadline))) break;
                tc_fence_after();
                const uint32_t sa = s0 + s * stage_bytes;
                const uint64_t da0 = sdesc_sw128(sa, 16, 1024);
                const uint64_t da1 = sdesc_sw128(sa + kTTileW, 16, 1024);
                const uint64_t dx = sdesc_sw128(sa + 2 * kTTileW, 16, 1024);
#pragma unroll
                for (int kk = 0; kk < kGemmBK / 16; ++kk) {
                    const uint32_t acc = (ks > ks0 || kk > 0) ? 1u : 0u;
                    umma_bf16(tbase, da0 + 2 * kk, dx + 2 * kk, id, acc);
                    if (two) umma_bf16(tbase + 256, da1 + 2 * kk, dx + 2 * kk, id, acc);
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
        // ------------------------------------------------------------ epilogue (warps 2..5)
        // Thread = W row (TMEM lane); each 32-column TMEM load holds 32 rows of
        // X for it.  The values go to shared memory as one output row per X
        // row (the stage ring is free once the last MMA has completed), then
        // one lane per warp copies whole rows out with bulk stores: a few
        // large writes per row instead of one 128-byte store per warp and X
        // row, which left the kernel's completion waiting long after its
        // last instruction.
        const int quad = warp & 3;
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        const int r = quad * 32 + lane;
        const int chunks = (p.M + 31) / 32;
        const bool ok = __all_sync(0xffffffffu, g_wait(acc_full, 0, deadline));
        if (ok) {
            tc_fence_after();
            if (p.act) {
                __nv_bfloat16* stage = reinterpret_cast<__nv_bfloat16*>(sm);  // [M][128]
#pragma unroll 1
                for (int c = 0; c < chunks; ++c) {
                    float g[32], u[32];
                    tmem_ld32(tbase + lane_off + 32 * c, g);
                    tmem_ld32(tbase + lane_off + 256 + 32 * c, u);
                    tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int t = 32 * c + j;
                        if (t < p.M) {
                            // gate and up are rounded to bf16 first, as when
                            // they are stored between kernels
                            const float gb = __bfloat162float(__float2bfloat16_rn(g[j]));
                            const float ub = __bfloat162float(__float2bfloat16_rn(u[j]));
                            stage[t * 128 + r] = __float2bfloat16_rn(silu_times(gb, ub));
                        }
                    }
                }
                fence_proxy_async_smem();
                epi_bar();
                if (lane == 0) {
                    const uint32_t bytes = static_cast<uint32_t>(nv0) * 2;
                    for (int t = quad; t < p.M; t += 4)
                        bulk_store(p.act + static_cast<size_t>(t) * p.paired_I + 128 * tile, stage + t * 128, bytes);
                    bulk_commit();
                    bulk_wait();
                }
            } else {
                float* stage = reinterpret_cast<float*>(sm);  // [M][128]
                for (int b = 0; b < (two ? 2 : 1); ++b) {
#pragma unroll 1
                    for (int c = 0; c < chunks; ++c) {
                        float v[32];
                        tmem_ld32(tbase + lane_off + 256 * b + 32 * c, v);
                        tmem_ld_wait();
#pragma unroll
                        for (int j = 0; j < 32; ++j) {
                            const int t = 32 * c + j;
                            if (t < p.M) stage[t * 128 + r] = v[j];
                        }
                    }
                    fence_proxy_async_smem();
                    epi_bar();
                    if (lane == 0) {
                        const uint32_t bytes = static_cast<uint32_t>(b ? nv1 : nv0) * 4;
                        float* dst = p.partials + static_cast<size_t>(split) * p.M * p.Nw + (b ? wb1 : wb0);
                        for (int t = quad; t < p.M; t += 4)
                            bulk_store(dst + static_cast<size_t>(t) * p.Nw, stage + t * 128, bytes);
                        bulk_commit();
                        bulk_wait();  // the stage is rewritten for the next block
                    }
                    epi_bar();
                }
            }
        } else {
            fail(8);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tbase, 512);
}

}  // namespace

GemmPlan gemm_plan(int M, int N, int K, int sms)
{
    GemmPlan g{};
    g.n_tiles = (N + kGemmBN - 1) / kGemmBN;
    g.m_pairs = (M + 2 * kGemmBM - 1) / (2 * kGemmBM);
    g.k_steps = (K + kGemmBK - 1) / kGemmBK;
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
    return cudaFuncSetAttribute(gemm_bf16_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, kGAlloc);
}

cudaError_t launch_gemm(const CUtensorMap& tm_x, const CUtensorMap& tm_w, const GemmParams& p,
                        int sms, cudaStream_t st)
{
    if (p.units <= 0) return cudaSuccess;
    const int grid = p.units < sms ? p.units : sms;
    if (p.splits == 1) {
        gemm_bf16_tc<<<grid, kGThreads, kGAlloc, st>>>(tm_x, tm_w, p);
        return cudaGetLastError();
    }
    // split K: the splits of a tile wait for one another, so every unit's CTA
    // must be resident at once (units <= SMs, one CTA per SM)
    if (p.units > sms) return cudaErrorInvalidConfiguration;
    CUtensorMap a = tm_x, b = tm_w;
    GemmParams q = p;
    void* args[] = {&a, &b, &q};
    return cudaLaunchCooperativeKernel(reinterpret_cast<const void*>(gemm_bf16_tc), dim3(grid),
                                       dim3(kGThreads), args, kGAlloc, st);
}

ThinPlan thin_plan(int M, int Nw, int K, int sms, int paired_I)
{
    ThinPlan g{};
    g.Mp = (M + 15) / 16 * 16;
    g.tiles = paired_I > 0 ? (paired_I + 127) / 128 : (Nw + 255) / 256;
    g.k_steps = (K + kGemmBK - 1) / kGemmBK;
    // split K while the tiles alone leave SMs idle, into as many ranges as
    // keep every unit in one wave
    int splits = g.tiles >= sms ? 1 : sms / g.tiles;
    splits = splits < 1 ? 1 : (splits > g.k_steps ? g.k_steps : splits);
    g.kps = (g.k_steps + splits - 1) / splits;
    g.splits = (g.k_steps + g.kps - 1) / g.kps;
    g.units = g.tiles * g.splits;
    const int sb = thin_stage_bytes(g.Mp);
    g.stages = (kTSmemMax - 1024 - kTBarBytes) / sb;
    g.stages = g.stages > kTMaxStages ? kTMaxStages : g.stages;
    g.smem = static_cast<size_t>(g.stages) * sb + kTBarBytes + 1024;
    g.partial_bytes = (paired_I > 0 && g.splits == 1) ? 0 : static_cast<size_t>(g.splits) * M * Nw * 4;
    return g;
}

cudaError_t thin_prepare()
{
    return cudaFuncSetAttribute(gemm_thin_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, kTSmemMax);
}

cudaError_t launch_thin_gemm(const CUtensorMap& tm_x, const CUtensorMap& tm_w, const ThinParams& p,
                             size_t smem, cudaStream_t st)
{
    const int units = (p.paired_I > 0 ? (p.paired_I + 127) / 128 : (p.Nw + 255) / 256) * p.splits;
    if (units <= 0) return cudaSuccess;
    if (p.M < 1 || p.M > kThinMaxRows || p.Mp != (p.M + 15) / 16 * 16 || p.stages < 2 ||
        p.stages > kTMaxStages || (p.act && (p.paired_I <= 0 || p.splits != 1)) || (!p.act && !p.partials) ||
        (p.paired_I > 0 ? (p.paired_I & 7) : (p.Nw & 3)) != 0 ||
        static_cast<size_t>(p.M) * 128 * 4 > static_cast<size_t>(p.stages) * thin_stage_bytes(p.Mp) ||
        smem > static_cast<size_t>(kTSmemMax) ||
        static_cast<size_t>(p.stages) * thin_stage_bytes(p.Mp) + kTBarBytes + 1024 > smem)
        return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(units);
    cfg.blockDim = dim3(kGThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, gemm_thin_tc, tm_x, tm_w, p);
}

}  // namespace statekv
