// K1: frame attention with saved log-sum-exp and fused importance partials.
//
// A work unit is 128 query rows of one KV-head group of one (stream, layer).
// Rows are packed token-major, row r = t * G + g (query head hkv*G + g of
// token t), so a tile covers ~128/G consecutive tokens and the in-frame
// causal mask of Eq. 5 skips every frame-key tile beyond its last token.
//
// Keys are the valid state slots (tiles of 128 from the compressed state)
// followed by the frame's tokens.  Two passes over the key tiles (App. B.1):
//   pass A  S = Q K^T  -> online max / sum per row -> log-sum-exp
//   pass B  S = Q K^T  -> P = exp(S - LSE) (fp32) -> column sums of P over the
//           tile's 128 rows (Eq. 1's importance, restricted to these rows) and
//           O += P V with P in bf16.
// tcgen05 runs every contraction with the A operand in TMEM (Q for Q K^T, P
// for P V), so each MMA streams only K or V from shared memory.  TMEM
// (512 columns): Q | P | S0 | S1 | O (layout below).
//
// K and V tiles stream through a ring of six 32 KB shared-memory slots in one
// sequence, pass A's K tiles, then pass B's K(0) V(0) K(1) V(1) ...; a slot is
// refilled once the MMAs that read it have completed (their commit arrives on
// the slot's barrier).
//
// The kernel is persistent: one CTA per SM walks work units (query tile, KV
// head, unit) in a fixed stride.  Ring, TMEM and barriers carry over from one
// unit to the next, so the producer loads the next unit's first tiles while
// the current one finishes, the next unit's Q goes into TMEM as soon as the
// last P V completes, and its first Q K^T run while the previous O is read out.
//
// 384 threads, three warpgroups:
//   WG0  warp 0 producer (TMA), warps 1 and 3 MMA issuers X and Y (warp 1
//        also owns TMEM), warp 2 the pass-B column-sum reducer.  tcgen05.mma
//        issue blocks at the tensor core's pace, so each barrier wait of an
//        issuing thread idles the tensor core; with two issuers one waits
//        while the other's MMAs run.  X issues the pass-A Q K^T of even tiles
//        and every pass-B Q K^T; Y the pass-A Q K^T of odd tiles and every
//        P V (in order, so O accumulates deterministically).  Descriptors are precomputed words, so an MMA
//        costs the issuing warp an add or two besides itself.
//   WG1, WG2  softmax warpgroups.  Pass A: thread = query row; they take
//        alternate key tiles, so the tensor core works on one warpgroup's
//        tile while the other computes exponentials.  Pass B: both work on
//        every tile, warpgroup w on keys [64 w, 64 w + 64), so each tile's P
//        is ready after half a tile's work.
// The column sums add a thread's rows in registers; the reducer warp adds the
// four warps' staged values per lane, then the lanes by a shuffle
// reduce-scatter, and writes the tile's importance partials.
// Every mbarrier wait is bounded by the watchdog; on expiry the CTA records
// DEV_TIMEOUT_ATTN, drains its in-flight copies and MMAs, frees TMEM and exits.
#include "sm103_ptx.cuh"
#include "statekv_kernels.cuh"

namespace statekv {
namespace {

using namespace ptx;

constexpr int kThreads = 384;
constexpr int kSlots = 6;        // 32 KB K/V tile slots (D = 128), one ring
// TMEM columns: Q [0, 64) | P [64, 128) | S0 | S1 | O; pass A also uses O's
// columns as a third score buffer S2.  Pass B puts even tiles' scores in S0
// and odd tiles' in S1.  P (bf16 pairs) of even tiles goes to the P buffer,
// so Q K^T can refill S0 as soon as both warpgroups have read the scores; P
// of odd tiles overwrites the scores it came from (each warpgroup the first
// 32 columns of its own 64), so Q K^T into S1 waits for the P V that reads
// it.  (TMEM has no room for a second P buffer next to Q, two score buffers
// and O.)
constexpr uint32_t kColP = 64;
constexpr uint32_t kColS0 = 128;
constexpr uint32_t kColS1 = 256;
constexpr uint32_t kColO = 384;
constexpr int kSA = 3;           // pass-A score buffers
// Pass-A barriers are indexed by tile mod 6 (buffer tile % 3, warpgroup and
// issuer tile % 2), so each waiter has seen the barrier's previous phase and
// can never mistake a phase two back for the one it waits for.
constexpr int kSA2 = 2 * kSA;

template <int D>
struct AttnLayout {
    static constexpr int kTileBytes = kBN * D * 2;  // one K or V tile
    static constexpr int kOffSlots = 0;
    // column-sum staging of one pass-B tile: float[2 wg][4 quadrants][4 chunks][32 lanes][4]
    static constexpr int kOffStage = kOffSlots + kSlots * kTileBytes;
    static constexpr int kOffStat = kOffStage + 2 * 4 * 4 * 32 * 4 * 4;  // float[5][128]
    static constexpr int kOffBar = kOffStat + 5 * kBM * 4;
    // slot_full[6] slot_empty[6] sa_full[6] sa_read[6] sb_full[2] sb_read[2]
    // p_full[2] pv_done[2] q_full o_full drain a_done a_read stage_full stage_free
    // o_read stall
    static constexpr int kNumBars = 41;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;
    static constexpr int kBytes = kOffMisc + 16;
    static constexpr int kAlloc = kBytes + 1024;  // room to align the base to 1 KB
    static_assert(kOffSlots % 1024 == 0 && kTileBytes % 1024 == 0, "align");
    static_assert(kAlloc <= 232448, "shared memory budget");
};

__device__ __forceinline__ float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float max3(float a, float b, float c)
{
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// Packed pair of floats in one 64-bit register (sm_100+ f32x2 arithmetic).
struct f2 {
    uint64_t r;
};

__device__ __forceinline__ f2 pk(float lo, float hi)
{
    f2 o;
    asm("mov.b64 %0, {%1, %2};" : "=l"(o.r) : "f"(lo), "f"(hi));
    return o;
}

__device__ __forceinline__ void upk(f2 x, float& lo, float& hi)
{
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(x.r));
}

__device__ __forceinline__ f2 fma2(f2 a, f2 b, f2 c)
{
    f2 d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d.r) : "l"(a.r), "l"(b.r), "l"(c.r));
    return d;
}

__device__ __forceinline__ f2 add2(f2 a, f2 b)
{
    f2 d;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d.r) : "l"(a.r), "l"(b.r));
    return d;
}

__device__ __forceinline__ unsigned long long globaltimer()
{
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Bounded wait on an mbarrier phase: polls until `deadline` (globaltimer ns).
__device__ __forceinline__ bool wait_until(uint64_t* bar, uint32_t parity,
                                           unsigned long long deadline)
{
    for (;;) {
#pragma unroll 1
        for (int i = 0; i < 64; ++i)
            if (mbar_try_wait(bar, parity)) return true;
        if (globaltimer() > deadline) return false;
    }
}

__device__ __forceinline__ void named_bar_sync(int id, int nthreads)
{
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

__device__ __forceinline__ void named_bar_arrive(int id, int nthreads)
{
    asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// One MMA group, D[d] (+)= A[a + 8k (+ kGapA when k >= NK/2)] * B_k for k < NK
// (bf16 in, fp32 accumulator, A in TMEM), with B's descriptor for step k given as its two
// 32-bit words (lo + off(k), hi): the issuing warp shares its SM sub-partition
// with the softmax warps, so each MMA should cost it as few instructions as
// possible.
template <int NK, bool kMajorB, uint32_t kGapA = 0>
__device__ __forceinline__ void mma_group(uint32_t d, uint32_t a, uint32_t blo, uint32_t bhi,
                                          uint32_t idesc, bool accumulate)
{
#pragma unroll
    for (int k = 0; k < NK; ++k) {
        // K-major B: 16 KB per 64-wide K half of a 128-row tile, 32 B per
        // 16-element step inside a half; MN-major B: 2 KB per step.
        const uint32_t off =
            kMajorB ? ((k >> 2) * (kBN * 128) + (k & 3) * 32) >> 4 : (k * 2048) >> 4;
        if (k == 0 && !accumulate)
            asm volatile(
                "{\n\t.reg .b64 bd;\n\t"
                "mov.b64 bd, {%2, %3};\n\t"
                "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], bd, %4, 0;\n\t}" ::"r"(d),
                "r"(a), "r"(blo + off), "r"(bhi), "r"(idesc)
                : "memory");
        else
            asm volatile(
                "{\n\t.reg .b64 bd;\n\t"
                "mov.b64 bd, {%2, %3};\n\t"
                "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], bd, %4, 1;\n\t}" ::"r"(d),
                "r"(a + 8 * k + (k >= NK / 2 ? kGapA : 0u)), "r"(blo + off), "r"(bhi), "r"(idesc)
                : "memory");
    }
}

// 16 consecutive 32-bit TMEM columns of this thread's lane <- registers.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0],"
        " {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
        "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
        "r"(r[15])
        : "memory");
}

__device__ __forceinline__ void tmem_st_wait()
{
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// 16 TMEM lanes x 64 columns -> 32 registers (.16x256b layout): register
// 4r + 2k + e holds lane (base + t/4 + 8k), column 8r + 2(t%4) + e, r < 8.
__device__ __forceinline__ void tmem_ld_16x256b_x8(uint32_t taddr, float (&v)[32])
{
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.16x256b.x8.b32"
        " {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15,"
        " %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31},"
        " [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// 16 registers -> 16 TMEM lanes x 32 columns (.16x128b layout): register
// 2r + k goes to lane (base + t/4 + 8k), column 4r + t%4, r < 8.
__device__ __forceinline__ void tmem_st_16x128b_x8(uint32_t taddr, const uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.st.sync.aligned.16x128b.x8.b32 [%0],"
        " {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
        "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
        "r"(r[15])
        : "memory");
}

// Sums over the 8 lanes that share lane % 4 (lane bits 2..4) of 32 values,
// as a reduce-scatter: lane l returns the sums of values 4 (l/4) .. +3.
__device__ __forceinline__ void lane8_reduce_scatter(float (&x)[32], int lane, float (&out)[4])
{
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        const bool up = (lane & 16) != 0;
        const float send = up ? x[i] : x[i + 16];
        const float keep = up ? x[i + 16] : x[i];
        x[i] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const bool up = (lane & 8) != 0;
        const float send = up ? x[i] : x[i + 8];
        const float keep = up ? x[i + 8] : x[i];
        x[i] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const bool up = (lane & 4) != 0;
        const float send = up ? x[i] : x[i + 4];
        const float keep = up ? x[i + 4] : x[i];
        out[i] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
    }
}

// One work unit: the 128 query rows of tile mt of KV head hkv of the call's
// unit u, with the key range the unit sees.  Units are numbered with the tile
// fastest, then the KV head, then the unit.
struct WorkUnit {
    int mt, hkv, u, ua;
    int count;  // visible keys before the frame (state slots or cache rows)
    int nst;    // key tiles over them
    int nft;    // frame key tiles the tile's last row can see
    int nt;     // nst + nft
    int rot;    // first state tile (see state_tile)
    int full_state;  // state tiles [0, full_state) hold 128 valid keys wherever they start
};

__device__ __forceinline__ WorkUnit work_unit(const AttnParams& p, int w)
{
    WorkUnit x;
    x.mt = w % p.MT;
    const int r = w / p.MT;
    x.hkv = r % p.Hkv;
    x.u = r / p.Hkv;
    x.ua = p.units.unit_abs(x.u);
    const int head = x.ua * p.Hkv + x.hkv;
    x.count = p.count_mul * ((p.B > 0 || p.count_mul > 1) ? p.counts[head] : 0) +
              (p.count_add ? p.count_add[head] : 0);
    x.nst = (x.count + kBN - 1) / kBN;
    const int row_hi = min(p.G * p.T, (x.mt + 1) * kBM) - 1;
    x.nft = p.causal ? (row_hi / p.G) / kBN + 1 : (p.T + kBN - 1) / kBN;
    x.nt = x.nst + x.nft;
    // The query tiles of one KV head read the same state tiles; each starts at
    // a different one (a fixed rotation) so they do not all request the same
    // L2 lines at the same moment.  Frame tiles keep their order.
    x.rot = x.nst > 0 ? (x.mt * 3) % x.nst : 0;
    // with a rotation the ragged state tile (the last one, if count % 128 != 0)
    // can come at any position; only when every state tile is whole is the
    // check skipped for all of them
    x.full_state = (x.count % kBN == 0) ? x.nst : 0;
    return x;
}

__device__ __forceinline__ int state_tile(const WorkUnit& x, int t)
{
    return t + x.rot < x.nst ? t + x.rot : t + x.rot - x.nst;
}

// Persistent: one CTA per SM walks the work units w = blockIdx.x, + gridDim.x,
// ...  The ring, the TMEM allocation and every barrier live across units: the
// producer loads the next unit's first tiles while the current one finishes,
// and the per-tile barrier phases continue from unit to unit (tb below counts
// the key tiles of the CTA's earlier units, so tile it of pass A is global
// tile tb + it, and item i of the ring is global item 3 tb + i).
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    frame_attn_lse_importance(const __grid_constant__ CUtensorMap tm_sk,
                              const __grid_constant__ CUtensorMap tm_sv,
                              const __grid_constant__ CUtensorMap tm_fk,
                              const __grid_constant__ CUtensorMap tm_fv, const AttnParams p)
{
    using L = AttnLayout<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
    uint8_t* sSlot = sm + L::kOffSlots;
    float4* stage = reinterpret_cast<float4*>(sm + L::kOffStage);
    float* stat = reinterpret_cast<float*>(sm + L::kOffStat);
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + L::kOffBar);
    uint64_t* slot_full = bars + 0;
    uint64_t* slot_empty = bars + 6;
    uint64_t* sa_full = bars + 12;  // pass A: Q K^T of global tile g done (index g % 6)
    uint64_t* sa_read = bars + 18;  // pass A: global tile g read by its warpgroup (index g % 6)
    uint64_t* sb_full = bars + 24;  // pass B: Q K^T of global tile g in score buffer g & 1
    uint64_t* sb_read = bars + 26;  // pass B: both warpgroups have read S0 ([1] unused)
    uint64_t* p_full = bars + 28;   // pass B: both warpgroups have written P of tile g (g & 1)
    uint64_t* pv_done = bars + 30;  // pass B: P V of tile g has completed (index g & 1)
    uint64_t* q_full = bars + 32;   // per unit: Q is in TMEM
    uint64_t* o_full = bars + 33;   // per unit: every P V has completed
    uint64_t* drain = bars + 34;
    uint64_t* a_done = bars + 35;   // per unit: every pass-A MMA has completed
    uint64_t* a_read = bars + 36;   // per unit: both warpgroups have read every pass-A tile
    uint64_t* stage_full = bars + 37;  // pass B: the tile's column sums are staged
    uint64_t* stage_free = bars + 38;  // pass B: the reducer warp has read them
    uint64_t* o_read = bars + 39;   // per unit: O has been read out of TMEM
    uint64_t* stall = bars + 40;    // watchdog self-test: never completed
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + L::kOffMisc);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(sm + L::kOffMisc + 4);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int T = p.T, G = p.G, B = p.B;
    const int rows = G * T;
    const int W = p.MT * p.Hkv * p.U;
    const int w0 = blockIdx.x, wstep = gridDim.x;

    // A softmax thread's Q row of unit w (thread 128 + i: warpgroup i / 128 - 1,
    // row i % 128; warpgroup wg holds d in [64 wg, 64 wg + 64)).
    uint4 qreg[8];
    auto load_q = [&](int w) {
        const int mt = w % p.MT, r = w / p.MT, hkv = r % p.Hkv, u = r / p.Hkv;
        const int tq = static_cast<int>(threadIdx.x) - 128;
        const int qwg = tq >> 7, qrow = tq & 127, qr = mt * kBM + qrow;
        const bool loads = p.q != nullptr && w < W && tq >= 0 && qwg * 64 < D && qr < rows;
        const int t = loads ? qr / G : 0, g = loads ? qr - t * G : 0;
        const uint4* src = reinterpret_cast<const uint4*>(
            p.q + ((static_cast<size_t>(loads ? u : 0) * T + t) * p.Hq + (loads ? hkv : 0) * G + g) * D +
            (loads ? qwg * 64 : 0));
#pragma unroll
        for (int i = 0; i < 8; ++i) qreg[i] = loads ? src[i] : make_uint4(0u, 0u, 0u, 0u);
    };
    // the first unit's rows load while the barriers and TMEM are set up
    load_q(w0);

    if (threadIdx.x == 0) {
        for (int i = 0; i < kSlots; ++i) {
            mbar_init(&slot_full[i], 1);
            mbar_init(&slot_empty[i], 1);
        }
        for (int i = 0; i < kSA2; ++i) {
            mbar_init(&sa_full[i], 1);
            mbar_init(&sa_read[i], 128);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&sb_full[i], 1);
            mbar_init(&sb_read[i], 256);
            mbar_init(&p_full[i], 256);
            mbar_init(&pv_done[i], 1);
        }
        mbar_init(a_read, 256);
        mbar_init(stage_full, 256);
        mbar_init(stage_free, 32);
        mbar_init(q_full, 256);
        mbar_init(o_full, 1);
        mbar_init(o_read, 256);
        mbar_init(drain, 2);   // one commit per MMA issuer
        mbar_init(a_done, 2);
        mbar_init(stall, 1);
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

    // Records an expired wait: DEV_TIMEOUT_ATTN with the waiting site in bits
    // 8..15 (see DeviceError), and tells every role to stop.
    auto fail = [&](int site) {
        if (atomicExch(const_cast<int*>(abort_flag), 1) == 0)  // first failure in the CTA
            *reinterpret_cast<volatile int32_t*>(p.status) = DEV_TIMEOUT_ATTN | (site << 8);
    };

    if (warp < 4) {
        asm volatile("setmaxnreg.dec.sync.aligned.u32 96;" ::: "memory");
        if (warp == 0) {
            // ------------------------------------------------------------ producer
            // One ring of tiles for both passes of every unit: per unit, pass A's
            // K tiles, then pass B's K(0) V(0) K(1) V(1) ...
            if (lane == 0) {
                tma_prefetch_desc(&tm_fk);
                tma_prefetch_desc(&tm_fv);
                if (B > 0) {
                    tma_prefetch_desc(&tm_sk);
                    tma_prefetch_desc(&tm_sv);
                }
                int last_use[kSlots];
#pragma unroll
                for (int sl = 0; sl < kSlots; ++sl) last_use[sl] = -1;
                bool ok = true;
                // the self-test's wait gives up at half the watchdog, so it is
                // deterministically the first wait of the launch to expire
                if (p.selftest_stall && !wait_until(stall, 0, globaltimer() + p.watchdog_ns / 2)) {
                    fail(1);
                    ok = false;
                }
                int n = 0;  // global item
                for (int w = w0; ok && w < W; w += wstep) {
                    const WorkUnit x = work_unit(p, w);
                    const unsigned long long deadline = globaltimer() + p.watchdog_ns;
                    for (int i = 0; i < 3 * x.nt; ++i, ++n) {
                        if (*abort_flag) {
                            ok = false;
                            break;
                        }
                        const int slot = n % kSlots, use = n / kSlots;
                        if (use >= 1 && !wait_until(&slot_empty[slot], (use - 1) & 1, deadline)) {
                            fail(2);
                            ok = false;
                            break;
                        }
                        const bool is_v = i >= x.nt && ((i - x.nt) & 1);
                        const int tile = i < x.nt ? i : (i - x.nt) >> 1;
                        const bool st = tile < x.nst;
                        const CUtensorMap* map = st ? (is_v ? &tm_sv : &tm_sk) : (is_v ? &tm_fv : &tm_fk);
                        const int c1 = st ? state_tile(x, tile) * kBN : x.hkv;
                        const int c2 = st ? x.hkv : (tile - x.nst) * kBN;
                        const int c3 = st ? x.ua : x.u;
                        uint8_t* dst = sSlot + slot * L::kTileBytes;
                        mbar_arrive_expect_tx(&slot_full[slot], L::kTileBytes);
#pragma unroll
                        for (int h = 0; h < D / 64; ++h)
                            tma_load_4d(dst + h * (kBN * 128), map, &slot_full[slot], h * 64, c1, c2, c3);
                        last_use[slot] = use;
                    }
                }
                const unsigned long long dl = globaltimer() + p.watchdog_ns;
                if (ok) {
                    // every slot's last tile has been read by its MMAs
                    for (int sl = 0; sl < kSlots; ++sl)
                        if (last_use[sl] >= 0) wait_until(&slot_empty[sl], last_use[sl] & 1, dl);
                } else {
                    // let copies already in flight land before the CTA's memory goes away
                    for (int sl = 0; sl < kSlots; ++sl)
                        if (last_use[sl] >= 0) wait_until(&slot_full[sl], last_use[sl] & 1, dl);
                }
            }
            __syncwarp();
        } else if (warp == 2) {
            // ------------------------------------------------------------ column-sum reducer
            // Pass B, per tile: the softmax threads stage their 16 row-summed
            // values (4 rows each); lane L adds the 4 quadrants' values of
            // staging lane L, then the 8 lanes that share L % 4 reduce-scatter
            // 32 values, leaving lane L with columns 64 wg + 16 jj + 8 h + 2 (L % 4) + e
            // (wg = m / 4, jj = m % 4, m = L / 4; h, e in {0, 1}).
            bool ok = true;
            int tb = 0;
            for (int w = w0; ok && w < W && p.partials != nullptr; w += wstep) {
                const WorkUnit x = work_unit(p, w);
                const unsigned long long deadline = globaltimer() + p.watchdog_ns;
                float* part = p.partials + ((static_cast<size_t>(x.u) * p.Hkv + x.hkv) * p.MT + x.mt) * p.P;
                for (int j = 0; j < x.nt; ++j) {
                    const int g = tb + j;
                    ok = __all_sync(0xffffffffu, wait_until(stage_full, g & 1, deadline));
                    if (!ok) {
                        if (lane == 0) fail(13);
                        break;
                    }
                    float xs[32];  // index (wg * 4 + jj) * 4 + i
#pragma unroll
                    for (int w2 = 0; w2 < 2; ++w2)
#pragma unroll
                        for (int jj = 0; jj < 4; ++jj) {
                            float4 a = stage[((w2 * 4 + 0) * 4 + jj) * 32 + lane];
#pragma unroll
                            for (int q = 1; q < 4; ++q) {
                                const float4 b4 = stage[((w2 * 4 + q) * 4 + jj) * 32 + lane];
                                a.x += b4.x;
                                a.y += b4.y;
                                a.z += b4.z;
                                a.w += b4.w;
                            }
                            const int o = (w2 * 4 + jj) * 4;
                            xs[o] = a.x;
                            xs[o + 1] = a.y;
                            xs[o + 2] = a.z;
                            xs[o + 3] = a.w;
                        }
                    mbar_arrive(stage_free);  // the softmax threads may stage the next tile
                    float sum4[4];
                    lane8_reduce_scatter(xs, lane, sum4);
                    const int m4 = lane >> 2, cbase = 64 * (m4 >> 2) + 16 * (m4 & 3) + 2 * (lane & 3);
                    const bool is_state = j < x.nst;
                    const int kb = (is_state ? state_tile(x, j) : j - x.nst) * kBN;
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int key = kb + cbase + 8 * (i >> 1) + (i & 1);
                        if (is_state ? key < x.count : key < T) part[is_state ? key : B + key] = sum4[i];
                    }
                }
                tb += x.nt;
            }
        } else if (warp == 1 || warp == 3) {
            // ------------------------------------------------------------ MMA issuers
            if (lane == 0) {
                const bool isx = warp == 1;
                const uint32_t aSlot = smem_addr(sSlot);
                const uint64_t dk = sdesc_sw128(aSlot, 16, 1024);         // K-major, slot 0
                const uint64_t dv = sdesc_sw128(aSlot, kBN * 128, 1024);  // MN-major, slot 0
                const uint32_t dk_lo = static_cast<uint32_t>(dk), d_hi = static_cast<uint32_t>(dk >> 32);
                const uint32_t dv_lo = static_cast<uint32_t>(dv);
                constexpr uint32_t kSlotStep = L::kTileBytes >> 4;  // descriptor address units
                const uint32_t tQ = tbase, tO = tbase + kColO;
                const uint32_t tS0 = tbase + kColS0, tS1 = tbase + kColS1;
                constexpr uint32_t kIdQK = idesc_bf16_f32(kBM, kBN, false, false);
                constexpr uint32_t kIdPV = idesc_bf16_f32(kBM, D, false, true);
                int site = 4;  // first wait that expired, for the status word
                bool ok = true;
                int tb = 0, k = 0;
                unsigned long long deadline = 0;
                // S = Q K^T of one tile into buffer tS; its slot is released by the commit
                auto qk = [&](int item, uint32_t tS, uint64_t* done) {
                    const int slot = item % kSlots;
                    tc_fence_after();
                    mma_group<D / 16, true>(tS, tQ, dk_lo + slot * kSlotStep, d_hi, kIdQK, false);
                    umma_commit(done);
                    umma_commit(&slot_empty[slot]);
                };
                for (int w = w0; ok && w < W; w += wstep, ++k) {
                    const WorkUnit x = work_unit(p, w);
                    deadline = globaltimer() + p.watchdog_ns;
                    const int nb = 3 * tb;  // the unit's first ring item
                    site = 4;
                    ok = wait_until(q_full, k & 1, deadline);
                    // pass A: X takes the even global tiles, Y the odd ones; buffer
                    // g % 3 (S0, S1, or O's columns, free once the previous unit's O
                    // has been read out)
                    for (int it = (isx ? 0 : 1) ^ (tb & 1); ok && it < x.nt; it += 2) {
                        const int g = tb + it, item = nb + it;
                        site = 5;
                        if (!(ok = wait_until(&slot_full[item % kSlots], (item / kSlots) & 1, deadline)))
                            break;
                        site = 6;
                        const int b = g % kSA;
                        if (g >= kSA && !(ok = wait_until(&sa_read[(g - kSA) % kSA2],
                                                          ((g - kSA) / kSA2) & 1, deadline)))
                            break;
                        if (b == 2 && it < kSA && k >= 1 &&
                            !(ok = wait_until(o_read, (k - 1) & 1, deadline)))
                            break;
                        qk(item, b == 0 ? tS0 : b == 1 ? tS1 : tO, &sa_full[g % kSA2]);
                    }
                    if (ok) umma_commit(a_done);
                    if (isx) {
                        // Pass B Q K^T, in tile order.  Every pass-A MMA has completed
                        // (so every pass-A load has landed: a slot's earlier occupant
                        // may have been the other issuer's) and both warpgroups have
                        // read every pass-A tile (the first tiles reuse S0 and S1).
                        if (ok) {
                            site = 9;
                            ok = wait_until(a_done, k & 1, deadline) && wait_until(a_read, k & 1, deadline);
                        }
                        for (int j = 0; ok && j < x.nt; ++j) {
                            const int g = tb + j, item = nb + x.nt + 2 * j, b = g & 1;
                            site = 5;
                            if (!(ok = wait_until(&slot_full[item % kSlots], (item / kSlots) & 1, deadline)))
                                break;
                            // the buffer's previous tile (g - 2) is consumed: read by both
                            // warpgroups (S0: its P went to the P buffer), or read by its
                            // P V (S1: its P overwrote the scores)
                            site = 6;
                            if (g >= 2 && !(ok = b == 0 ? wait_until(&sb_read[0], ((g - 2) >> 1) & 1, deadline)
                                                        : wait_until(&pv_done[1], ((g - 2) >> 1) & 1, deadline)))
                                break;
                            qk(item, b ? tS1 : tS0, &sb_full[b]);
                        }
                    } else {
                        // O += P(j) V(j): P of even global tiles in the P buffer (keys
                        // 0..63 then 64..127), of odd ones over S1 (keys 0..63 at its
                        // columns 0..31, keys 64..127 at 64..95)
                        for (int j = 0; ok && j < x.nt; ++j) {
                            const int g = tb + j, item = nb + x.nt + 2 * j + 1, b = g & 1;
                            const int slot = item % kSlots;
                            // the V tile usually landed long ago: its wait goes first, so
                            // the wait that P ends is the last before the MMAs
                            site = 8;
                            if (!(ok = wait_until(&slot_full[slot], (item / kSlots) & 1, deadline))) break;
                            site = 7;
                            if (!(ok = wait_until(&p_full[b], (g >> 1) & 1, deadline))) break;
                            tc_fence_after();
                            if (b == 0)
                                mma_group<kBN / 16, false>(tO, tbase + kColP, dv_lo + slot * kSlotStep,
                                                           d_hi, kIdPV, j > 0);
                            else
                                mma_group<kBN / 16, false, 32>(tO, tS1, dv_lo + slot * kSlotStep, d_hi,
                                                               kIdPV, j > 0);
                            umma_commit(&pv_done[b]);
                            umma_commit(&slot_empty[slot]);
                        }
                        if (ok) umma_commit(o_full);
                    }
                    tb += x.nt;
                }
                if (!ok) fail(site + (isx ? 0 : 16));
                // Every MMA issued so far must finish before TMEM is released.
                umma_commit(drain);
                wait_until(drain, 0, globaltimer() + p.watchdog_ns);
            }
            __syncwarp();
        }
        tc_fence_before();
        __syncthreads();
        if (warp == 1) tmem_dealloc(tbase, 512);
    } else {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 200;" ::: "memory");
        // ------------------------------------------------------------ softmax warpgroups
        const int wg = (warp >> 2) - 1;          // 0 or 1
        const int quad = warp & 3;               // TMEM lane quadrant of this warp
        const int row = quad * 32 + lane;        // TMEM lane = query row of the tile
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        const float c = p.scale_log2;
        const int cq = 2 * (lane & 3);           // this thread's column offset in 8
        const int c0 = 64 * wg;                  // this warpgroup's first key of a tile
        const uint32_t tSh0 = tbase + lane_off + kColS0 + c0;   // this warpgroup's S0 half
        const uint32_t tSh1 = tbase + lane_off + kColS1 + c0;   // its S1 half (and odd P)
        const uint32_t tPh = tbase + lane_off + kColP + c0 / 2;  // its even-tile P
        float4* mystage = stage + (wg * 4 + quad) * 4 * 32 + lane;  // chunk jj at + jj * 32
        float* nl_row = stat + 4 * kBM;  // -lse of every row of the tile
        const f2 cc = pk(c, c);

        // O rows of unit x -> bf16 out; warpgroup wg stores columns [wg D/2, (wg+1) D/2)
        auto store_o = [&](const WorkUnit& x) {
            const int my_r = x.mt * kBM + row;
            __nv_bfloat16* dst = p.out;
            if (my_r < rows) {
                const int t = my_r / G, g = my_r - t * G;
                dst += ((static_cast<size_t>(x.u) * T + t) * p.Hq + x.hkv * G + g) * D;
            }
#pragma unroll
            for (int cc2 = 0; cc2 < D / 64; ++cc2) {
                const int col = wg * (D / 2) + cc2 * 32;
                float o[32];
                tmem_ld32(tbase + lane_off + kColO + col, o);
                tmem_ld_wait();
                if (my_r < rows) {
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const uint4 v4 = make_uint4(
                            pack_bf16x2(o[e * 8 + 0], o[e * 8 + 1]), pack_bf16x2(o[e * 8 + 2], o[e * 8 + 3]),
                            pack_bf16x2(o[e * 8 + 4], o[e * 8 + 5]), pack_bf16x2(o[e * 8 + 6], o[e * 8 + 7]));
                        *reinterpret_cast<uint4*>(dst + col + e * 8) = v4;
                    }
                }
            }
        };

        bool ok = true;
        int site = 10;  // first wait that expired, for the status word
        int tb = 0, k = 0;
        WorkUnit prev{};
        for (int w = w0; ok && w < W; w += wstep, ++k) {
            const WorkUnit x = work_unit(p, w);
            const unsigned long long deadline = globaltimer() + p.watchdog_ns;
            const int my_r = x.mt * kBM + row;
            const bool row_valid = my_r < rows;
            const int my_tq = row_valid ? my_r / G : T;  // padding rows see every frame key

            {   // Q row -> TMEM columns [0, D/2) (bf16 pairs); warpgroup wg stores
                // d in [64 wg, 64 wg + 64) when D = 128, warpgroup 0 all of D = 64.
                // Every Q K^T of the previous unit has completed (its P V have).
                if (wg * 64 < D) {
                    uint32_t w32[32];
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        w32[4 * i] = qreg[i].x;
                        w32[4 * i + 1] = qreg[i].y;
                        w32[4 * i + 2] = qreg[i].z;
                        w32[4 * i + 3] = qreg[i].w;
                    }
                    tmem_st16(tbase + lane_off + wg * 32, *reinterpret_cast<uint32_t(*)[16]>(&w32[0]));
                    tmem_st16(tbase + lane_off + wg * 32 + 16,
                              *reinterpret_cast<uint32_t(*)[16]>(&w32[16]));
                    tmem_st_wait();
                }
                tc_fence_before();
                mbar_arrive(q_full);
            }
            if (k >= 1) {  // the previous unit's O, while this unit's first Q K^T run
                store_o(prev);
                tc_fence_before();
                mbar_arrive(o_read);
            }

            // ---------------- pass A: online max / sum of exp2 over this warpgroup's tiles
            float m = -INFINITY, l = 0.f;  // log2 units, scaled
            const int it0 = wg ^ (tb & 1);  // this warpgroup takes the global tiles of parity wg
            for (int it = it0; it < x.nt; it += 2) {
                const int g = tb + it;
                const int b = g % kSA;  // score buffer of this tile
                ok = __all_sync(0xffffffffu, wait_until(&sa_full[g % kSA2], (g / kSA2) & 1, deadline));
                if (!ok) break;
                tc_fence_after();
                const uint32_t tSa = tbase + lane_off + (b == 0 ? kColS0 : b == 1 ? kColS1 : kColO);
                int lim;  // keys [0, lim) of this tile are visible to this row
                if (it < x.nst) {
                    lim = min(kBN, x.count - state_tile(x, it) * kBN);
                } else {
                    const int f0 = (it - x.nst) * kBN;
                    lim = min(kBN, (p.causal ? min(T, my_tq + 1) : T) - f0);
                }
                // the whole tile into registers, then release the buffer at once so
                // the next Q K^T into it can start while this one is reduced
                float v[4][32];
#pragma unroll
                for (int ch = 0; ch < 4; ++ch) tmem_ld32(tSa + ch * 32, v[ch]);
                tmem_ld_wait();
                tc_fence_before();
                mbar_arrive(&sa_read[g % kSA2]);
                // after its last tile is in registers, this thread holds no pass-A
                // score buffer: pass B's Q K^T may start while the sums finish
                if (it + 2 >= x.nt) mbar_arrive(a_read);
                if (lim < kBN) {
#pragma unroll
                    for (int ch = 0; ch < 4; ++ch)
#pragma unroll
                        for (int e = 0; e < 32; ++e)
                            v[ch][e] = (ch * 32 + e < lim) ? v[ch][e] : -INFINITY;
                }
                float mx[4];
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) mx[q4] = fmaxf(v[q4][0], v[q4][1]);
#pragma unroll
                for (int ch = 0; ch < 4; ++ch)
#pragma unroll
                    for (int e = 2; e < 32; e += 2)
                        mx[ch] = max3(mx[ch], v[ch][e], v[ch][e + 1]);
                const float m_new =
                    fmaxf(m, fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * c);  // c > 0
                if (m_new != -INFINITY) {
                    const f2 nm = pk(-m_new, -m_new);
                    f2 acc[4] = {pk(0.f, 0.f), pk(0.f, 0.f), pk(0.f, 0.f), pk(0.f, 0.f)};
#pragma unroll
                    for (int ch = 0; ch < 4; ++ch)
#pragma unroll
                        for (int e = 0; e < 32; e += 2) {
                            float x0, x1;
                            upk(fma2(pk(v[ch][e], v[ch][e + 1]), cc, nm), x0, x1);
                            acc[(e >> 1) & 3] = add2(acc[(e >> 1) & 3], pk(ex2(x0), ex2(x1)));
                        }
                    float s0, s1;
                    upk(add2(add2(acc[0], acc[1]), add2(acc[2], acc[3])), s0, s1);
                    l = l * ex2(m - m_new) + (s0 + s1);
                    m = m_new;
                }
            }
            if (it0 >= x.nt) mbar_arrive(a_read);  // a warpgroup without pass-A tiles
            // The pass-A -> pass-B hand-over exchanges the row statistics through
            // two named barriers (1, then 2).  A warp whose pass-A wait expired
            // records it, arrives at both barriers without waiting and leaves: the
            // other warpgroup may have no pass-A tile left to wait on and be at
            // barrier 1 already, and it is released through both; its pass-B waits
            // then expire, since every pass-B step needs both warpgroups.  (An
            // AND-reducing barrier that both leave together measured 5.8% slower
            // over the whole launch.)
            if (!ok) {
                fail(10 + 32 * wg);  // Q K^T in pass A
                named_bar_arrive(1, 256);
                named_bar_arrive(2, 256);
                break;
            }
            stat[(wg * 2 + 0) * kBM + row] = m;
            stat[(wg * 2 + 1) * kBM + row] = l;
            named_bar_sync(1, 256);
            site = 11;
            float nlse;  // -log2-sum-exp of this row (scaled); -inf for padding rows
            {
                const float m0 = stat[0 * kBM + row], l0 = stat[1 * kBM + row];
                const float m1 = stat[2 * kBM + row], l1 = stat[3 * kBM + row];
                const float mm = fmaxf(m0, m1);
                const float ll = l0 * ex2(m0 - mm) + l1 * ex2(m1 - mm);
                nlse = row_valid ? -(mm + __log2f(ll)) : -INFINITY;
            }
            if (wg == 0) nl_row[row] = nlse;
            named_bar_sync(2, 256);
            float nl4[4];  // -lse of this thread's 4 rows, index 2h + k
            int tq4[4];    // token of each row (T for padding rows)
#pragma unroll
            for (int h = 0; h < 2; ++h)
#pragma unroll
                for (int k2 = 0; k2 < 2; ++k2) {
                    const int rr = quad * 32 + 16 * h + lane / 4 + 8 * k2;
                    nl4[2 * h + k2] = nl_row[rr];
                    const int gr = x.mt * kBM + rr;
                    tq4[2 * h + k2] = gr < rows ? gr / G : T;
                }
            // the next unit's Q rows load during pass B
            load_q(w + wstep);

            // ---------------- pass B: P = exp2(S c - lse) -> TMEM (bf16) and column sums
            // Both warpgroups work on every tile, warpgroup wg on its keys
            // [64 wg, 64 wg + 64), so a tile's P is ready after half a tile's work.
            // TMEM is read in 16-lane x 256-bit groups: a thread holds 4 rows
            // (quadrant rows 16h + t/4 + 8k, h, k in {0, 1}) x 16 columns
            // (8r + 2(t%4) + e).  P of even global tiles goes to the P buffer (so
            // Q K^T can refill S0 once both warpgroups have read it); P of odd
            // tiles overwrites the first half of this warpgroup's own S1 columns
            // (Q K^T into S1 waits for that P V).
            float* part = p.partials ? p.partials + ((static_cast<size_t>(x.u) * p.Hkv + x.hkv) * p.MT + x.mt) * p.P
                                     : nullptr;
            site = 12;
            for (int j = 0; ok && j < x.nt; ++j) {
                const int g = tb + j, b = g & 1;
                ok = __all_sync(0xffffffffu, wait_until(&sb_full[b], (g >> 1) & 1, deadline));
                if (!ok) break;
                tc_fence_after();
                int lim4[4] = {kBN, kBN, kBN, kBN};  // keys [0, lim) of this tile are visible to each row
                bool full = true;
                if (j >= x.full_state) {  // the last state tile or a frame tile
                    if (j < x.nst) {
                        const int lim = min(kBN, x.count - state_tile(x, j) * kBN);
#pragma unroll
                        for (int q4 = 0; q4 < 4; ++q4) lim4[q4] = lim;
                    } else {
                        const int f0 = (j - x.nst) * kBN;
#pragma unroll
                        for (int q4 = 0; q4 < 4; ++q4)
                            lim4[q4] = min(kBN, (p.causal ? min(T, tq4[q4] + 1) : T) - f0);
                    }
                    const int lmin = min(min(lim4[0], lim4[1]), min(lim4[2], lim4[3]));
                    full = lmin >= c0 + 64;
                }
                float v[2][32];
#pragma unroll
                for (int h = 0; h < 2; ++h) tmem_ld_16x256b_x8((b ? tSh1 : tSh0) + ((16u * h) << 16), v[h]);
                tmem_ld_wait();
                if (b == 0) {
                    tc_fence_before();
                    mbar_arrive(&sb_read[0]);  // Q K^T of tile g + 2 may overwrite S0
                }
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int r = 0; r < 8; ++r)
#pragma unroll
                        for (int k2 = 0; k2 < 2; ++k2) {
                            const int i = 4 * r + 2 * k2;
                            const float nk = nl4[2 * h + k2];
                            float x0, x1;
                            upk(fma2(pk(v[h][i], v[h][i + 1]), cc, pk(nk, nk)), x0, x1);
                            v[h][i] = ex2(x0);
                            v[h][i + 1] = ex2(x1);
                        }
                if (!full) {  // a ragged tile: keys at or past a row's limit get zero weight
#pragma unroll
                    for (int h = 0; h < 2; ++h)
#pragma unroll
                        for (int r = 0; r < 8; ++r)
#pragma unroll
                            for (int k2 = 0; k2 < 2; ++k2) {
                                const int i = 4 * r + 2 * k2;
                                const int col = c0 + 8 * r + cq, lim = lim4[2 * h + k2];
                                v[h][i] = col < lim ? v[h][i] : 0.f;
                                v[h][i + 1] = col + 1 < lim ? v[h][i + 1] : 0.f;
                            }
                }
                // the P buffer is free once the P V of tile g - 2 has read it
                if (b == 0 && g >= 2)
                    ok = __all_sync(0xffffffffu, wait_until(&pv_done[0], ((g - 2) >> 1) & 1, deadline));
                if (!ok) break;
                tc_fence_after();
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    uint32_t pw[16];  // register 2r + k: row k, P column 4r + t%4
#pragma unroll
                    for (int r = 0; r < 8; ++r)
#pragma unroll
                        for (int k2 = 0; k2 < 2; ++k2)
                            pw[2 * r + k2] = pack_bf16x2(v[h][4 * r + 2 * k2], v[h][4 * r + 2 * k2 + 1]);
                    tmem_st_16x128b_x8((b ? tSh1 : tPh) + ((16u * h) << 16), pw);
                }
                tmem_st_wait();
                tc_fence_before();
                mbar_arrive(&p_full[b]);
                // the column sums run while the tensor core does this tile's P V:
                // value 2r + e is column 8r + cq + e summed over the thread's rows;
                // the reducer warp adds them across lanes and warps
                if (part != nullptr) {
                    float cs[16];
#pragma unroll
                    for (int r = 0; r < 8; ++r) {
                        const f2 a = add2(pk(v[0][4 * r], v[0][4 * r + 1]), pk(v[0][4 * r + 2], v[0][4 * r + 3]));
                        const f2 bb = add2(pk(v[1][4 * r], v[1][4 * r + 1]), pk(v[1][4 * r + 2], v[1][4 * r + 3]));
                        upk(add2(a, bb), cs[2 * r], cs[2 * r + 1]);
                    }
                    if (g >= 1)  // the reducer has read the previous tile's values
                        ok = __all_sync(0xffffffffu, wait_until(stage_free, (g - 1) & 1, deadline));
                    if (!ok) break;
#pragma unroll
                    for (int jj = 0; jj < 4; ++jj)
                        mystage[jj * 32] = make_float4(cs[4 * jj], cs[4 * jj + 1], cs[4 * jj + 2], cs[4 * jj + 3]);
                    mbar_arrive(stage_full);
                }
            }
            if (!ok) break;
            // Frame keys no row of this tile can see receive zero importance here.
            if (part != nullptr)
                for (int t = x.nft * kBN + (threadIdx.x - 128); t < T; t += 256) part[B + t] = 0.f;
            // every P V of the unit has completed: O is final, and TMEM's Q and
            // score columns are free for the next unit
            site = 14;
            ok = __all_sync(0xffffffffu, wait_until(o_full, k & 1, deadline));
            if (!ok) break;
            tc_fence_after();
            prev = x;
            tb += x.nt;
        }
        if (ok && k >= 1) store_o(prev);  // the last unit's O
        if (!ok) fail(site + 32 * wg);
        tc_fence_before();
        __syncthreads();
    }
}

// The register split (WG0 down to 96, the softmax warpgroups up to 200 per
// thread) must fit the registers the CTA is launched with, or setmaxnreg.inc
// would wait forever: 128 * 96 + 256 * 200 = 63488 <= 384 threads * 168.
constexpr int kLaunchRegs = 168;
static_assert(128 * 96 + 256 * 200 <= kThreads * kLaunchRegs, "register split");

// SMs of each device, read by attn_prepare with that device current; the
// persistent grid of a launch is sized for the device current at the launch.
constexpr int kMaxDevices = 64;
int g_num_sms[kMaxDevices] = {};

int current_device_sms()
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 1;
    return g_num_sms[dev] > 0 ? g_num_sms[dev] : 1;
}

template <int D>
cudaError_t prepare_one()
{
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, frame_attn_lse_importance<D>);
    if (e != cudaSuccess) return e;
    if (fa.numRegs < kLaunchRegs) return cudaErrorInvalidConfiguration;
    int dev = 0, sms = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    g_num_sms[dev] = sms;
    return cudaFuncSetAttribute(frame_attn_lse_importance<D>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                AttnLayout<D>::kAlloc);
}

// One CTA per SM (at most one per work unit); each walks its units in order.
template <int D>
cudaError_t launch_one(const CUtensorMap& tm_sk, const CUtensorMap& tm_sv, const CUtensorMap& tm_fk,
                       const CUtensorMap& tm_fv, const AttnParams& p0, int U, cudaStream_t st)
{
    AttnParams p = p0;
    p.U = U;
    const long long W = static_cast<long long>(p.MT) * p.Hkv * U;
    if (W <= 0) return cudaSuccess;
    if (W > 0x7FFFFFFFll) return cudaErrorInvalidValue;
    const int sms = current_device_sms();
    const int grid = static_cast<int>(W < sms ? W : sms);
    frame_attn_lse_importance<D><<<grid, kThreads, AttnLayout<D>::kAlloc, st>>>(tm_sk, tm_sv, tm_fk,
                                                                              tm_fv, p);
    return cudaSuccess;
}

}  // namespace

int device_sm_count() { return current_device_sms(); }

size_t attn_smem_bytes(int D)
{
    return D == 64 ? AttnLayout<64>::kAlloc : AttnLayout<128>::kAlloc;
}

cudaError_t attn_prepare(int D)
{
    return D == 64 ? prepare_one<64>() : prepare_one<128>();
}

cudaError_t launch_attn(int D, const CUtensorMap& tm_sk, const CUtensorMap& tm_sv,
                        const CUtensorMap& tm_fk, const CUtensorMap& tm_fv, const AttnParams& p,
                        int U, cudaStream_t st)
{
    const cudaError_t e = D == 64 ? launch_one<64>(tm_sk, tm_sv, tm_fk, tm_fv, p, U, st)
                                  : launch_one<128>(tm_sk, tm_sv, tm_fk, tm_fv, p, U, st);
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace statekv
