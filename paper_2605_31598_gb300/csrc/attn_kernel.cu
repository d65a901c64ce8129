// K1: frame attention with saved log-sum-exp and fused importance partials.
//
// One CTA owns 128 query rows of one KV-head group of one (stream, layer).
// Rows are packed token-major, row r = t * G + g (query head hkv*G + g of
// token t), so a tile covers ~128/G consecutive tokens and the in-frame
// causal mask of Eq. 5 skips every frame-key tile beyond its last token.
//
// Keys are the valid state slots (tiles of 128 from the compressed state)
// followed by the frame's tokens.  Two passes over the key tiles (App. B.1):
//   pass A  S = Q K^T          (M = queries)  -> online max / sum -> LSE per row
//   pass B  S^T = K Q^T        (M = keys)     -> P = exp(S - LSE) in fp32;
//           thread = key, so the column sum over the tile's queries (Eq. 1's
//           importance, restricted to these rows) is a register sum;
//           O += P V           (P bf16, MN-major from shared memory)
// Both contractions run on tcgen05 with fp32 accumulators in TMEM.  K and V
// tiles arrive by TMA (128-byte swizzle) in four 32 KB shared-memory slots:
// pass A streams K through all four; pass B streams K through slots 0-1 and
// V through slots 2-3, loaded by two independent producer threads so a V
// slot that is still waiting for its P.V never holds back the next K load.
//
// 384 threads, three warpgroups:
//   WG0  warp 0 K producer, warp 1 TMEM owner + MMA issuer, warp 2 V
//        producer (warp 3 idle)
//   WG1, WG2  softmax / importance warpgroups; they take alternate key tiles,
//        so while one works on tile j the other works on j+1 and the tensor
//        core computes j+2 (three TMEM score buffers + the O accumulator fill
//        the 512 TMEM columns).
// The per-element work uses packed f32x2 FMA/ADD, three-input max and
// independent accumulators so no dependency chain runs the length of a tile.
// Every mbarrier wait is bounded by the watchdog; on expiry the CTA records
// DEV_TIMEOUT_ATTN, drains its in-flight copies and MMAs, frees TMEM and exits.
#include "sm103_ptx.cuh"
#include "statekv_kernels.cuh"

namespace statekv {
namespace {

using namespace ptx;

constexpr int kThreads = 384;
constexpr int kSBuf = 3;  // TMEM score buffers

template <int D>
struct AttnLayout {
    static constexpr int kQBytes = kBM * D * 2;
    static constexpr int kTileBytes = kBN * D * 2;  // one K or V tile
    static constexpr int kPBytes = kBM * kBN * 2;
    static constexpr int kOffQ = 0;
    static constexpr int kOffSlots = kOffQ + kQBytes;          // 4 K/V tile slots
    static constexpr int kOffP = kOffSlots + 4 * kTileBytes;
    static constexpr int kOffNLse = kOffP + 2 * kPBytes;   // float[128]: -LSE*log2e per row
    static constexpr int kOffTq = kOffNLse + kBM * 4;      // int[128]: token of each row
    static constexpr int kOffBar = kOffTq + kBM * 4;
    // slot_full[4] slot_empty[4] s_full[3] s_empty[3] p_full[2] p_empty[2]
    // q_full o_full drain a_done
    static constexpr int kNumBars = 22;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;
    static constexpr int kBytes = kOffMisc + 16;
    static constexpr int kAlloc = kBytes + 1024;  // room to align the base to 1 KB
    static_assert(kOffSlots % 1024 == 0 && kOffP % 1024 == 0, "align");
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

// K-major SW128 operand with `rows` rows: k-step ks (16 elements) of the tile.
__device__ __forceinline__ uint64_t kmajor_desc(uint32_t base, int ks, int rows)
{
    return sdesc_sw128(base + (ks >> 2) * (rows * 128) + (ks & 3) * 32, 16, 1024);
}

// MN-major SW128 operand whose 64-wide MN blocks are `block_bytes` apart:
// k-step ks covers 16 K rows (2 groups of 8).
__device__ __forceinline__ uint64_t mnmajor_desc(uint32_t base, int ks, uint32_t block_bytes)
{
    return sdesc_sw128(base + ks * 2048, block_bytes, 1024);
}

__device__ __forceinline__ float4 lds_f4(const void* p)
{
    // volatile: re-read per tile instead of being hoisted out of the tile
    // loop (keeping 128 per-column values live would exhaust registers)
    float4 v;
    asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(smem_addr(p)));
    return v;
}

__device__ __forceinline__ int4 lds_i4(const void* p)
{
    int4 v;
    asm volatile("ld.shared.v4.s32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(smem_addr(p)));
    return v;
}

// Pass A tile `it` occupies slot it % 4; pass B K tile j occupies slot j % 2
// and V tile j slot 2 + j % 2.  The use count of a slot before pass B is the
// number of pass-A tiles it held.
__device__ __forceinline__ int pass_a_uses(int nt, int slot)
{
    return nt > slot ? (nt - slot + 3) / 4 : 0;
}

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
    uint8_t* sQ = sm + L::kOffQ;
    uint8_t* sSlot = sm + L::kOffSlots;
    uint8_t* sP = sm + L::kOffP;
    float* nlse2 = reinterpret_cast<float*>(sm + L::kOffNLse);
    int* tq = reinterpret_cast<int*>(sm + L::kOffTq);
    // (m, l) of both softmax warpgroups at the end of pass A: float[2][2][128].
    // It borrows the P buffers, which are first written after the merge.
    float* stat = reinterpret_cast<float*>(sm + L::kOffP);
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + L::kOffBar);
    uint64_t* slot_full = bars + 0;
    uint64_t* slot_empty = bars + 4;
    uint64_t* s_full = bars + 8;
    uint64_t* s_empty = bars + 11;
    uint64_t* p_full = bars + 14;
    uint64_t* p_empty = bars + 16;
    uint64_t* q_full = bars + 18;
    uint64_t* o_full = bars + 19;
    uint64_t* drain = bars + 20;
    uint64_t* a_done = bars + 21;  // every pass-A MMA has completed
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + L::kOffMisc);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(sm + L::kOffMisc + 4);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int mt = blockIdx.x;
    const int hkv = blockIdx.y;
    const int u = blockIdx.z;
    const int ua = p.units.unit_abs(u);
    const int T = p.T, G = p.G, B = p.B;
    const int rows = G * T;
    const int count = (B > 0) ? p.counts[ua * p.Hkv + hkv] : 0;
    const int nst = (count + kBN - 1) / kBN;
    const int row_hi = min(rows, (mt + 1) * kBM) - 1;
    const int nft = p.causal ? (row_hi / G) / kBN + 1 : (T + kBN - 1) / kBN;
    const int nt = nst + nft;
    const unsigned long long deadline = globaltimer() + p.watchdog_ns;

    if (threadIdx.x == 0) {
        for (int i = 0; i < 4; ++i) {
            mbar_init(&slot_full[i], 1);
            mbar_init(&slot_empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&p_full[i], 128);
            mbar_init(&p_empty[i], 1);
        }
        for (int i = 0; i < kSBuf; ++i) {
            mbar_init(&s_full[i], 1);
            mbar_init(&s_empty[i], 128);
        }
        mbar_init(q_full, 256);
        mbar_init(o_full, 1);
        mbar_init(drain, 1);
        mbar_init(a_done, 1);
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

    auto fail = [&]() {
        *abort_flag = 1;
        *reinterpret_cast<volatile int32_t*>(p.status) = DEV_TIMEOUT_ATTN;
    };

    if (warp < 4) {
        asm volatile("setmaxnreg.dec.sync.aligned.u32 80;" ::: "memory");
        if (warp == 0 || warp == 2) {
            // ------------------------------------------------------------ producers
            // warp 0: K tiles of both passes; warp 2: V tiles of pass B
            if (lane == 0) {
                const bool kprod = warp == 0;
                if (kprod) {
                    tma_prefetch_desc(&tm_fk);
                    if (B > 0) tma_prefetch_desc(&tm_sk);
                } else {
                    tma_prefetch_desc(&tm_fv);
                    if (B > 0) tma_prefetch_desc(&tm_sv);
                }
                const CUtensorMap* smap = kprod ? &tm_sk : &tm_sv;
                const CUtensorMap* fmap = kprod ? &tm_fk : &tm_fv;
                int last_use[4] = {-1, -1, -1, -1};
                // Slots 2-3 also carry pass-A K tiles: the V producer starts only
                // once every pass-A MMA has released them (before that, a wait on
                // their empty barriers could match an earlier phase of the same
                // parity).
                if (!kprod && !wait_until(a_done, 0, deadline)) fail();
                // loads: pass A (K producer only) then pass B
                const int nload = kprod ? 2 * nt : nt;
                for (int n = 0; n < nload; ++n) {
                    if (*abort_flag) break;
                    int slot, use, tile;
                    if (kprod && n < nt) {
                        tile = n;
                        slot = n & 3;
                        use = n >> 2;
                    } else {
                        tile = kprod ? n - nt : n;
                        slot = (kprod ? 0 : 2) + (tile & 1);
                        use = pass_a_uses(nt, slot) + (tile >> 1);
                    }
                    if (use >= 1 && !wait_until(&slot_empty[slot], (use - 1) & 1, deadline)) {
                        fail();
                        break;
                    }
                    uint8_t* dst = sSlot + slot * L::kTileBytes;
                    mbar_arrive_expect_tx(&slot_full[slot], L::kTileBytes);
#pragma unroll
                    for (int h = 0; h < D / 64; ++h) {
                        if (tile < nst)
                            tma_load_4d(dst + h * (kBN * 128), smap, &slot_full[slot], h * 64,
                                        tile * kBN, hkv, ua);
                        else
                            tma_load_4d(dst + h * (kBN * 128), fmap, &slot_full[slot], h * 64,
                                        hkv, (tile - nst) * kBN, u);
                    }
                    last_use[slot] = use;
                }
                if (*abort_flag) {
                    // Let copies already in flight land before the CTA's memory goes away.
                    const unsigned long long dl = globaltimer() + p.watchdog_ns;
                    for (int sl = 0; sl < 4; ++sl)
                        if (last_use[sl] >= 0) wait_until(&slot_full[sl], last_use[sl] & 1, dl);
                }
            }
            __syncwarp();
        } else if (warp == 1) {
            // ------------------------------------------------------------ MMA issuer
            if (lane == 0) {
                const uint32_t aQ = smem_addr(sQ), aSlot = smem_addr(sSlot), aP = smem_addr(sP);
                const uint32_t tO = tbase + kSBuf * 128;
                constexpr uint32_t kIdQK = idesc_bf16_f32(kBM, kBN, false, false);
                constexpr uint32_t kIdKQ = idesc_bf16_f32(kBN, kBM, false, false);
                constexpr uint32_t kIdPV = idesc_bf16_f32(kBM, D, true, true);
                bool ok = wait_until(q_full, 0, deadline);
                // score MMA of sequence index it (pass A: it < nt; pass B: nt + j)
                auto issue_s = [&](int it, bool transposed) -> bool {
                    const int b = it % kSBuf;
                    const int j = it - nt;
                    const int slot = transposed ? (j & 1) : (it & 3);
                    const int use = transposed ? pass_a_uses(nt, slot) + (j >> 1) : (it >> 2);
                    if (!wait_until(&slot_full[slot], use & 1, deadline)) return false;
                    if (it >= kSBuf && !wait_until(&s_empty[b], ((it / kSBuf) - 1) & 1, deadline))
                        return false;
                    tc_fence_after();
                    const uint32_t kb = aSlot + slot * L::kTileBytes;
                    const uint32_t tS = tbase + b * 128;
#pragma unroll
                    for (int k = 0; k < D / 16; ++k) {
                        if (transposed)
                            umma_bf16(tS, kmajor_desc(kb, k, kBN), kmajor_desc(aQ, k, kBM), kIdKQ, k > 0);
                        else
                            umma_bf16(tS, kmajor_desc(aQ, k, kBM), kmajor_desc(kb, k, kBN), kIdQK, k > 0);
                    }
                    umma_commit(&s_full[b]);
                    umma_commit(&slot_empty[slot]);
                    return true;
                };
                auto issue_pv = [&](int j) -> bool {
                    const int w = (nt + j) & 1, slot = 2 + (j & 1);
                    const int use = pass_a_uses(nt, slot) + (j >> 1);
                    if (!wait_until(&p_full[w], (j >> 1) & 1, deadline)) return false;
                    if (!wait_until(&slot_full[slot], use & 1, deadline)) return false;
                    tc_fence_after();
                    const uint32_t pbase = aP + w * L::kPBytes;
                    const uint32_t vbase = aSlot + slot * L::kTileBytes;
#pragma unroll
                    for (int k = 0; k < kBN / 16; ++k)
                        umma_bf16(tO, mnmajor_desc(pbase, k, kBN * 128),
                                  mnmajor_desc(vbase, k, kBN * 128), kIdPV, (j > 0 || k > 0));
                    umma_commit(&p_empty[w]);
                    umma_commit(&slot_empty[slot]);
                    return true;
                };
                for (int it = 0; ok && it < nt; ++it) ok = issue_s(it, false);  // pass A
                if (ok) umma_commit(a_done);
                for (int j = 0; ok && j < nt; ++j) {                             // pass B
                    ok = issue_s(nt + j, true);
                    if (ok && j >= 2) ok = issue_pv(j - 2);
                }
                if (ok && nt >= 2) ok = issue_pv(nt - 2);
                if (ok) ok = issue_pv(nt - 1);
                if (ok) umma_commit(o_full);
                if (!ok) fail();
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
        asm volatile("setmaxnreg.inc.sync.aligned.u32 208;" ::: "memory");
        // ------------------------------------------------------------ softmax warpgroups
        const int wg = (warp >> 2) - 1;          // 0 or 1
        const int ct = threadIdx.x - 128;        // 0..255 across both warpgroups
        const int quad = warp & 3;               // TMEM lane quadrant of this warp
        const int row = quad * 32 + lane;        // TMEM lane = tile row
        const uint32_t tlane = tbase + (static_cast<uint32_t>(quad * 32) << 16);
        const float c = p.scale_log2;

        for (int i = ct; i < kBM; i += 256) {
            const int r = mt * kBM + i;
            tq[i] = r < rows ? r / G : -1;
        }
        {   // Q tile -> K-major SW128 shared memory, zero rows past the group
            constexpr int kChunks = D / 8;  // 16-byte chunks per row
            const __nv_bfloat16* qu = p.q + static_cast<size_t>(u) * T * p.Hq * D;
            for (int idx = ct; idx < kBM * kChunks; idx += 256) {
                const int ri = idx / kChunks, ch = idx % kChunks;
                const int r = mt * kBM + ri;
                uint4 val = make_uint4(0, 0, 0, 0);
                if (r < rows) {
                    const int t = r / G, g = r - t * G;
                    val = *reinterpret_cast<const uint4*>(
                        qu + (static_cast<size_t>(t) * p.Hq + hkv * G + g) * D + ch * 8);
                }
                *reinterpret_cast<uint4*>(sQ + (ch >> 3) * (kBM * 128) + sw128_offset(ri, ch & 7)) =
                    val;
            }
        }
        fence_proxy_async_smem();
        mbar_arrive(q_full);

        bool ok = true;
        // ---------------- pass A: thread = query row; online max / sum of exp2
        const int my_r = mt * kBM + row;
        const int my_tq = my_r < rows ? my_r / G : T;  // padding rows see every frame key
        float m = -INFINITY, l = 0.f;                   // in log2 units, scaled
        for (int it = wg; it < nt; it += 2) {
            const int b = it % kSBuf;
            ok = __all_sync(0xffffffffu, wait_until(&s_full[b], (it / kSBuf) & 1, deadline));
            if (!ok) break;
            tc_fence_after();
            int lim;  // keys [0, lim) of this tile are visible to this row
            if (it < nst) {
                lim = min(kBN, count - it * kBN);
            } else {
                const int f0 = (it - nst) * kBN;
                lim = min(kBN, (p.causal ? min(T, my_tq + 1) : T) - f0);
            }
            // four 32-column chunks; the next chunk's TMEM load overlaps this
            // chunk's math (tcgen05.wait::ld waits for every load issued so far)
            float v[2][32];
            tmem_ld32(tlane + b * 128, v[0]);
            tmem_ld_wait();
#pragma unroll
            for (int ch = 0; ch < 4; ++ch) {
                float (&x)[32] = v[ch & 1];
                if (ch < 3) tmem_ld32(tlane + b * 128 + (ch + 1) * 32, v[(ch + 1) & 1]);
                if (lim < kBN) {
#pragma unroll
                    for (int j = 0; j < 32; ++j) x[j] = (ch * 32 + j < lim) ? x[j] : -INFINITY;
                }
                float mx[4];
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) mx[q4] = fmaxf(x[q4 * 2], x[q4 * 2 + 1]);
#pragma unroll
                for (int j = 8; j < 32; j += 8)
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4)
                        mx[q4] = max3(mx[q4], x[j + q4 * 2], x[j + q4 * 2 + 1]);
                const float m_new =
                    fmaxf(m, fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * c);  // c > 0
                if (m_new != -INFINITY) {
                    const f2 cc = pk(c, c), nm = pk(-m_new, -m_new);
                    f2 acc[4] = {pk(0.f, 0.f), pk(0.f, 0.f), pk(0.f, 0.f), pk(0.f, 0.f)};
#pragma unroll
                    for (int j = 0; j < 32; j += 2) {
                        float x0, x1;
                        upk(fma2(pk(x[j], x[j + 1]), cc, nm), x0, x1);
                        acc[(j >> 1) & 3] = add2(acc[(j >> 1) & 3], pk(ex2(x0), ex2(x1)));
                    }
                    float s0, s1;
                    upk(add2(add2(acc[0], acc[1]), add2(acc[2], acc[3])), s0, s1);
                    l = l * ex2(m - m_new) + (s0 + s1);
                    m = m_new;
                }
                if (ch < 3) tmem_ld_wait();
            }
            tc_fence_before();
            mbar_arrive(&s_empty[b]);
        }
        stat[(wg * 2 + 0) * kBM + row] = m;
        stat[(wg * 2 + 1) * kBM + row] = l;
        named_bar_sync(1, 256);
        if (wg == 0) {
            const float m0 = stat[0 * kBM + row], l0 = stat[1 * kBM + row];
            const float m1 = stat[2 * kBM + row], l1 = stat[3 * kBM + row];
            const float mm = fmaxf(m0, m1);
            const float ll = l0 * ex2(m0 - mm) + l1 * ex2(m1 - mm);
            nlse2[row] = (my_r < rows) ? -(mm + __log2f(ll)) : -INFINITY;
        }
        named_bar_sync(1, 256);

        // ---------------- pass B: thread = key; columns = the tile's query rows
        float* part = p.partials + ((static_cast<size_t>(u) * p.Hkv + hkv) * p.MT + mt) * p.P;
        const int t_lo = (mt * kBM) / G;  // first query token of the tile
        uint8_t* Pb = sP + wg * L::kPBytes;
        for (int j = (wg - nt) & 1; ok && j < nt; j += 2) {
            const int it = nt + j, b = it % kSBuf;
            ok = __all_sync(0xffffffffu, wait_until(&s_full[b], (it / kSBuf) & 1, deadline));
            if (!ok) break;
            tc_fence_after();
            float v[2][32];
            tmem_ld32(tlane + b * 128, v[0]);
            const bool is_state = j < nst;
            const int key = is_state ? j * kBN + row : (j - nst) * kBN + row;
            const bool kvalid = is_state ? key < count : key < T;
            // the tile needs a per-element causal test unless all of its keys
            // precede the tile's first query token
            const bool diag = !is_state && p.causal && ((j - nst) * kBN + kBN - 1 > t_lo);
            const f2 cc = pk(c, c);
            f2 acc[4] = {pk(0.f, 0.f), pk(0.f, 0.f), pk(0.f, 0.f), pk(0.f, 0.f)};
            uint32_t pp[kBM / 2];  // the tile's P row, bf16 pairs
            tmem_ld_wait();
#pragma unroll
            for (int ch = 0; ch < 4; ++ch) {
                float (&x)[32] = v[ch & 1];
                if (ch < 3) tmem_ld32(tlane + b * 128 + (ch + 1) * 32, v[(ch + 1) & 1]);
#pragma unroll
                for (int g8 = 0; g8 < 4; ++g8) {
                    const int c8 = ch * 4 + g8;  // columns 8*c8 .. 8*c8+7
                    const float4 la = lds_f4(&nlse2[c8 * 8]);
                    const float4 lb = lds_f4(&nlse2[c8 * 8 + 4]);
                    const f2 nl[4] = {pk(la.x, la.y), pk(la.z, la.w), pk(lb.x, lb.y),
                                      pk(lb.z, lb.w)};
                    float pr[8];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        float x0, x1;
                        upk(fma2(pk(x[g8 * 8 + 2 * e], x[g8 * 8 + 2 * e + 1]), cc, nl[e]), x0, x1);
                        pr[2 * e] = ex2(x0);
                        pr[2 * e + 1] = ex2(x1);
                    }
                    if (diag) {
                        const int4 qa = lds_i4(&tq[c8 * 8]);
                        const int4 qb = lds_i4(&tq[c8 * 8 + 4]);
                        const int qs[8] = {qa.x, qa.y, qa.z, qa.w, qb.x, qb.y, qb.z, qb.w};
#pragma unroll
                        for (int e = 0; e < 8; ++e) pr[e] = (qs[e] >= key) ? pr[e] : 0.f;
                    }
                    if (!kvalid) {
#pragma unroll
                        for (int e = 0; e < 8; ++e) pr[e] = 0.f;
                    }
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        acc[e] = add2(acc[e], pk(pr[2 * e], pr[2 * e + 1]));
                        pp[c8 * 4 + e] = pack_bf16x2(pr[2 * e], pr[2 * e + 1]);
                    }
                }
                if (ch < 3) tmem_ld_wait();
            }
            // the score buffer is free as soon as it is in registers
            tc_fence_before();
            mbar_arrive(&s_empty[b]);
            if (j >= 2) {
                ok = __all_sync(0xffffffffu,
                                wait_until(&p_empty[wg], ((j >> 1) - 1) & 1, deadline));
                if (!ok) break;
            }
#pragma unroll
            for (int c8 = 0; c8 < kBM / 8; ++c8)
                *reinterpret_cast<uint4*>(Pb + (c8 >> 3) * (kBN * 128) + sw128_offset(row, c8 & 7)) =
                    make_uint4(pp[c8 * 4], pp[c8 * 4 + 1], pp[c8 * 4 + 2], pp[c8 * 4 + 3]);
            fence_proxy_async_smem();
            mbar_arrive(&p_full[wg]);
            float s0, s1;
            upk(add2(add2(acc[0], acc[1]), add2(acc[2], acc[3])), s0, s1);
            if (kvalid) part[is_state ? key : B + key] = s0 + s1;
        }
        // Frame keys no row of this tile can see receive zero importance here.
        for (int t = nft * kBN + ct; t < T; t += 256) part[B + t] = 0.f;

        // ---------------- epilogue: O rows (thread = query row) -> bf16 out;
        // warpgroup wg stores columns [wg*D/2, (wg+1)*D/2)
        if (ok) ok = __all_sync(0xffffffffu, wait_until(o_full, 0, deadline));
        if (ok) {
            tc_fence_after();
            const bool valid = my_r < rows;
            __nv_bfloat16* dst = p.out;
            if (valid) {
                const int t = my_r / G, g = my_r - t * G;
                dst += ((static_cast<size_t>(u) * T + t) * p.Hq + hkv * G + g) * D;
            }
#pragma unroll
            for (int cc = 0; cc < D / 64; ++cc) {
                const int col = wg * (D / 2) + cc * 32;
                float o[32];
                tmem_ld32(tlane + kSBuf * 128 + col, o);
                tmem_ld_wait();
                if (valid) {
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const uint4 w = make_uint4(
                            pack_bf16x2(o[e * 8 + 0], o[e * 8 + 1]),
                            pack_bf16x2(o[e * 8 + 2], o[e * 8 + 3]),
                            pack_bf16x2(o[e * 8 + 4], o[e * 8 + 5]),
                            pack_bf16x2(o[e * 8 + 6], o[e * 8 + 7]));
                        *reinterpret_cast<uint4*>(dst + col + e * 8) = w;
                    }
                }
            }
        }
        if (!ok) fail();
        tc_fence_before();
        __syncthreads();
    }
}

}  // namespace

size_t attn_smem_bytes(int D)
{
    return D == 64 ? AttnLayout<64>::kAlloc : AttnLayout<128>::kAlloc;
}

// The register split (WG0 down to 80, the softmax warpgroups up to 208 per
// thread) must fit the registers the CTA is launched with, or setmaxnreg.inc
// would wait forever: 128 * 80 + 256 * 208 = 63488 <= 384 threads * 168.
constexpr int kLaunchRegs = 168;
static_assert(128 * 80 + 256 * 208 <= kThreads * kLaunchRegs, "register split");

template <int D>
cudaError_t prepare_one()
{
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, frame_attn_lse_importance<D>);
    if (e != cudaSuccess) return e;
    if (fa.numRegs < kLaunchRegs) return cudaErrorInvalidConfiguration;
    return cudaFuncSetAttribute(frame_attn_lse_importance<D>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                AttnLayout<D>::kAlloc);
}

cudaError_t attn_prepare(int D)
{
    return D == 64 ? prepare_one<64>() : prepare_one<128>();
}

cudaError_t launch_attn(int D, const CUtensorMap& tm_sk, const CUtensorMap& tm_sv,
                        const CUtensorMap& tm_fk, const CUtensorMap& tm_fv, const AttnParams& p,
                        int U, cudaStream_t st)
{
    const dim3 grid(p.MT, p.Hkv, U);
    if (D == 64)
        frame_attn_lse_importance<64>
            <<<grid, kThreads, AttnLayout<64>::kAlloc, st>>>(tm_sk, tm_sv, tm_fk, tm_fv, p);
    else
        frame_attn_lse_importance<128>
            <<<grid, kThreads, AttnLayout<128>::kAlloc, st>>>(tm_sk, tm_sv, tm_fk, tm_fv, p);
    return cudaGetLastError();
}

}  // namespace statekv
