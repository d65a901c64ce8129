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
// Both contractions run on tcgen05 with fp32 accumulators in TMEM; K and V
// tiles arrive by TMA (128-byte swizzle) through a two-stage ring.
//
// Warp roles (192 threads):  warp 0 TMA producer, warp 1 TMEM owner + MMA
// issuer, warps 2..5 softmax / importance / epilogue (one TMEM lane quadrant
// each).  Every mbarrier wait is bounded by the watchdog; on expiry the CTA
// records DEV_TIMEOUT_ATTN, drains its in-flight copies and MMAs, frees TMEM
// and exits.
#include "sm103_ptx.cuh"
#include "statekv_kernels.cuh"

#include <cfloat>

namespace statekv {
namespace {

using namespace ptx;

template <int D>
struct AttnLayout {
    static constexpr int kStages = 2;
    static constexpr int kQBytes = kBM * D * 2;
    static constexpr int kTileBytes = kBN * D * 2;  // one K or V tile
    static constexpr int kPBytes = kBM * kBN * 2;
    static constexpr int kOffQ = 0;
    static constexpr int kOffK = kOffQ + kQBytes;
    static constexpr int kOffV = kOffK + kStages * kTileBytes;
    static constexpr int kOffP = kOffV + kStages * kTileBytes;
    static constexpr int kOffLse = kOffP + 2 * kPBytes;
    static constexpr int kOffTq = kOffLse + kBM * 4;
    static constexpr int kOffBar = kOffTq + kBM * 4;
    // kv_full[2], kv_empty[2], s_full[2], s_empty[2], p_full[2], p_empty[2],
    // q_full, o_full, drain
    static constexpr int kNumBars = 15;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;
    static constexpr int kBytes = kOffMisc + 16;
    static constexpr int kAlloc = kBytes + 1024;  // room to align the base to 1 KB
    static_assert(kOffK % 1024 == 0 && kOffV % 1024 == 0 && kOffP % 1024 == 0, "align");
    static_assert(kAlloc <= 232448, "shared memory budget");
};

__device__ __forceinline__ float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
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

template <int D>
__global__ void __launch_bounds__(192, 1)
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
    uint8_t* sK = sm + L::kOffK;
    uint8_t* sV = sm + L::kOffV;
    uint8_t* sP = sm + L::kOffP;
    float* lse2 = reinterpret_cast<float*>(sm + L::kOffLse);
    int* tq = reinterpret_cast<int*>(sm + L::kOffTq);
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + L::kOffBar);
    uint64_t* kv_full = bars + 0;
    uint64_t* kv_empty = bars + 2;
    uint64_t* s_full = bars + 4;
    uint64_t* s_empty = bars + 6;
    uint64_t* p_full = bars + 8;
    uint64_t* p_empty = bars + 10;
    uint64_t* q_full = bars + 12;
    uint64_t* o_full = bars + 13;
    uint64_t* drain = bars + 14;
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
        for (int i = 0; i < 2; ++i) {
            mbar_init(&kv_full[i], 1);
            mbar_init(&kv_empty[i], 1);
            mbar_init(&s_full[i], 1);
            mbar_init(&s_empty[i], 128);
            mbar_init(&p_full[i], 128);
            mbar_init(&p_empty[i], 1);
        }
        mbar_init(q_full, 128);
        mbar_init(o_full, 1);
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

    auto fail = [&]() {
        *abort_flag = 1;
        *reinterpret_cast<volatile int32_t*>(p.status) = DEV_TIMEOUT_ATTN;
    };

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            tma_prefetch_desc(&tm_fk);
            tma_prefetch_desc(&tm_fv);
            if (B > 0) {
                tma_prefetch_desc(&tm_sk);
                tma_prefetch_desc(&tm_sv);
            }
            int issued = 0;
            for (int it = 0; it < 2 * nt; ++it) {
                if (*abort_flag) break;
                const int s = it % L::kStages;
                if (it >= L::kStages &&
                    !wait_until(&kv_empty[s], ((it / L::kStages) - 1) & 1, deadline)) {
                    fail();
                    break;
                }
                const bool pass_b = it >= nt;
                const int tile = pass_b ? it - nt : it;
                mbar_arrive_expect_tx(&kv_full[s], L::kTileBytes * (pass_b ? 2 : 1));
                uint8_t* dk = sK + s * L::kTileBytes;
                uint8_t* dv = sV + s * L::kTileBytes;
#pragma unroll
                for (int h = 0; h < D / 64; ++h) {
                    if (tile < nst) {
                        tma_load_4d(dk + h * (kBN * 128), &tm_sk, &kv_full[s], h * 64, tile * kBN,
                                    hkv, ua);
                        if (pass_b)
                            tma_load_4d(dv + h * (kBN * 128), &tm_sv, &kv_full[s], h * 64,
                                        tile * kBN, hkv, ua);
                    } else {
                        const int f0 = (tile - nst) * kBN;
                        tma_load_4d(dk + h * (kBN * 128), &tm_fk, &kv_full[s], h * 64, hkv, f0, u);
                        if (pass_b)
                            tma_load_4d(dv + h * (kBN * 128), &tm_fv, &kv_full[s], h * 64, hkv,
                                        f0, u);
                    }
                }
                issued = it + 1;
            }
            if (*abort_flag) {
                // Let copies already in flight land before the CTA's memory goes away.
                for (int it = max(0, issued - L::kStages); it < issued; ++it)
                    wait_until(&kv_full[it % L::kStages], (it / L::kStages) & 1,
                               globaltimer() + p.watchdog_ns);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t aQ = smem_addr(sQ), aK = smem_addr(sK), aV = smem_addr(sV),
                           aP = smem_addr(sP);
            const uint32_t tS[2] = {tbase, tbase + 128};
            const uint32_t tO = tbase + 256;
            constexpr uint32_t kIdQK = idesc_bf16_f32(kBM, kBN, false, false);
            constexpr uint32_t kIdKQ = idesc_bf16_f32(kBN, kBM, false, false);
            constexpr uint32_t kIdPV = idesc_bf16_f32(kBM, D, true, true);
            bool ok = wait_until(q_full, 0, deadline);
            // pass A: S = Q K^T
            for (int it = 0; ok && it < nt; ++it) {
                const int s = it % L::kStages, b = it & 1;
                ok = wait_until(&kv_full[s], (it / L::kStages) & 1, deadline);
                if (ok && it >= 2) ok = wait_until(&s_empty[b], ((it >> 1) - 1) & 1, deadline);
                if (!ok) break;
                tc_fence_after();
                const uint32_t kb = aK + s * L::kTileBytes;
#pragma unroll
                for (int ks = 0; ks < D / 16; ++ks)
                    umma_bf16(tS[b], kmajor_desc(aQ, ks, kBM), kmajor_desc(kb, ks, kBN), kIdQK,
                              ks > 0);
                umma_commit(&s_full[b]);
                umma_commit(&kv_empty[s]);
            }
            auto issue_pv = [&](int j) -> bool {
                const int it = nt + j, s = it % L::kStages, pb = j & 1;
                if (!wait_until(&p_full[pb], (j >> 1) & 1, deadline)) return false;
                tc_fence_after();
                const uint32_t pbase = aP + pb * L::kPBytes;
                const uint32_t vbase = aV + s * L::kTileBytes;
#pragma unroll
                for (int ks = 0; ks < kBN / 16; ++ks)
                    umma_bf16(tO, mnmajor_desc(pbase, ks, kBN * 128),
                              mnmajor_desc(vbase, ks, kBN * 128), kIdPV, (j > 0 || ks > 0));
                umma_commit(&p_empty[pb]);
                umma_commit(&kv_empty[s]);
                return true;
            };
            // pass B: S^T = K Q^T, then O += P V one tile behind
            for (int j = 0; ok && j < nt; ++j) {
                const int it = nt + j, s = it % L::kStages, b = it & 1;
                ok = wait_until(&kv_full[s], (it / L::kStages) & 1, deadline);
                if (ok && it >= 2) ok = wait_until(&s_empty[b], ((it >> 1) - 1) & 1, deadline);
                if (!ok) break;
                tc_fence_after();
                const uint32_t kb = aK + s * L::kTileBytes;
#pragma unroll
                for (int ks = 0; ks < D / 16; ++ks)
                    umma_bf16(tS[b], kmajor_desc(kb, ks, kBN), kmajor_desc(aQ, ks, kBM), kIdKQ,
                              ks > 0);
                umma_commit(&s_full[b]);
                if (j > 0) ok = issue_pv(j - 1);
            }
            if (ok) ok = issue_pv(nt - 1);
            if (ok) umma_commit(o_full);
            if (!ok) fail();
            // Every MMA issued so far must finish before TMEM is released.
            umma_commit(drain);
            wait_until(drain, 0, globaltimer() + p.watchdog_ns);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ softmax warps
        const int ct = threadIdx.x - 64;         // 0..127
        const int quad = warp & 3;               // TMEM lane quadrant of this warp
        const int row = quad * 32 + lane;        // TMEM lane = tile row
        const uint32_t tlane = tbase + (static_cast<uint32_t>(quad * 32) << 16);

        // Query tokens of the tile's rows (-1 for padding rows).
        for (int i = ct; i < kBM; i += 128) {
            const int r = mt * kBM + i;
            tq[i] = r < rows ? r / G : -1;
        }
        // Q tile -> K-major SW128 shared memory, zero rows past the group.
        {
            constexpr int kChunks = D / 8;  // 16-byte chunks per row
            const __nv_bfloat16* qu = p.q + static_cast<size_t>(u) * T * p.Hq * D;
            for (int idx = ct; idx < kBM * kChunks; idx += 128) {
                const int ri = idx / kChunks, ch = idx % kChunks;
                const int r = mt * kBM + ri;
                uint4 val = make_uint4(0, 0, 0, 0);
                if (r < rows) {
                    const int t = r / G, g = r - (r / G) * G;
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
        float m = -INFINITY, l = 0.f;
        for (int it = 0; it < nt; ++it) {
            const int b = it & 1;
            ok = __all_sync(0xffffffffu, wait_until(&s_full[b], (it >> 1) & 1, deadline));
            if (!ok) break;
            tc_fence_after();
            float v[kBN];
#pragma unroll
            for (int c = 0; c < kBN / 32; ++c)
                tmem_ld32(tlane + b * 128 + c * 32, *reinterpret_cast<float(*)[32]>(&v[c * 32]));
            tmem_ld_wait();
            tc_fence_before();
            mbar_arrive(&s_empty[b]);
            int lim;  // keys [0, lim) of this tile are visible to this row
            if (it < nst) {
                lim = min(kBN, count - it * kBN);
            } else {
                const int f0 = (it - nst) * kBN;
                lim = min(kBN, (p.causal ? min(T, my_tq + 1) : T) - f0);
            }
            float mx = -INFINITY;
#pragma unroll
            for (int c = 0; c < kBN; ++c) {
                v[c] = (c < lim) ? v[c] * p.scale_log2 : -INFINITY;
                mx = fmaxf(mx, v[c]);
            }
            const float m_new = fmaxf(m, mx);
            if (m_new != -INFINITY) {
                float sum = 0.f;
#pragma unroll
                for (int c = 0; c < kBN; ++c) sum += ex2(v[c] - m_new);
                l = l * ex2(m - m_new) + sum;
                m = m_new;
            }
        }
        lse2[row] = (my_r < rows) ? m + __log2f(l) : INFINITY;
        named_bar_sync(1, 128);

        // ---------------- pass B: thread = key; columns = the tile's query rows
        float* part = p.partials + ((static_cast<size_t>(u) * p.Hkv + hkv) * p.MT + mt) * p.P;
        for (int j = 0; ok && j < nt; ++j) {
            const int it = nt + j, b = it & 1, pb = j & 1;
            ok = __all_sync(0xffffffffu, wait_until(&s_full[b], (it >> 1) & 1, deadline));
            if (!ok) break;
            tc_fence_after();
            float v[kBM];
#pragma unroll
            for (int c = 0; c < kBM / 32; ++c)
                tmem_ld32(tlane + b * 128 + c * 32, *reinterpret_cast<float(*)[32]>(&v[c * 32]));
            tmem_ld_wait();
            tc_fence_before();
            mbar_arrive(&s_empty[b]);
            if (j >= 2) {
                ok = __all_sync(0xffffffffu,
                                wait_until(&p_empty[pb], ((j >> 1) - 1) & 1, deadline));
                if (!ok) break;
            }
            const bool is_state = j < nst;
            const int key = is_state ? j * kBN + row : (j - nst) * kBN + row;
            const bool kvalid = is_state ? key < count : key < T;
            const int thr = (!is_state && p.causal) ? key : 0;  // query token must be >= thr
            uint8_t* Pb = sP + pb * L::kPBytes;
            float colsum = 0.f;
#pragma unroll
            for (int c8 = 0; c8 < kBM / 8; ++c8) {
                const float4 la = *reinterpret_cast<const float4*>(&lse2[c8 * 8]);
                const float4 lb = *reinterpret_cast<const float4*>(&lse2[c8 * 8 + 4]);
                const int4 qa = *reinterpret_cast<const int4*>(&tq[c8 * 8]);
                const int4 qb = *reinterpret_cast<const int4*>(&tq[c8 * 8 + 4]);
                const float ls[8] = {la.x, la.y, la.z, la.w, lb.x, lb.y, lb.z, lb.w};
                const int qs[8] = {qa.x, qa.y, qa.z, qa.w, qb.x, qb.y, qb.z, qb.w};
                float pr[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const float x = ex2(fmaf(v[c8 * 8 + e], p.scale_log2, -ls[e]));
                    pr[e] = (kvalid && qs[e] >= thr) ? x : 0.f;
                    colsum += pr[e];
                }
                const uint4 w = make_uint4(pack_bf16x2(pr[0], pr[1]), pack_bf16x2(pr[2], pr[3]),
                                           pack_bf16x2(pr[4], pr[5]), pack_bf16x2(pr[6], pr[7]));
                *reinterpret_cast<uint4*>(Pb + (c8 >> 3) * (kBN * 128) +
                                          sw128_offset(row, c8 & 7)) = w;
            }
            fence_proxy_async_smem();
            mbar_arrive(&p_full[pb]);
            if (kvalid) part[is_state ? key : B + key] = colsum;
        }
        // Frame keys no row of this tile can see receive zero importance here.
        for (int t = nft * kBN + ct; t < T; t += 128) part[B + t] = 0.f;

        // ---------------- epilogue: O rows (thread = query row) -> bf16 out
        if (ok) ok = __all_sync(0xffffffffu, wait_until(o_full, 0, deadline));
        if (ok) {
            tc_fence_after();
            const bool valid = my_r < rows;
            __nv_bfloat16* dst = p.out;
            if (valid) {
                const int t = my_r / G, g = my_r - (my_r / G) * G;
                dst += ((static_cast<size_t>(u) * T + t) * p.Hq + hkv * G + g) * D;
            }
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                float o[32];
                tmem_ld32(tlane + 256 + c * 32, o);
                tmem_ld_wait();
                if (valid) {
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const uint4 w = make_uint4(
                            pack_bf16x2(o[e * 8 + 0], o[e * 8 + 1]),
                            pack_bf16x2(o[e * 8 + 2], o[e * 8 + 3]),
                            pack_bf16x2(o[e * 8 + 4], o[e * 8 + 5]),
                            pack_bf16x2(o[e * 8 + 6], o[e * 8 + 7]));
                        *reinterpret_cast<uint4*>(dst + c * 32 + e * 8) = w;
                    }
                }
            }
        }
        if (!ok) fail();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tbase, 512);
}

}  // namespace

size_t attn_smem_bytes(int D)
{
    return D == 64 ? AttnLayout<64>::kAlloc : AttnLayout<128>::kAlloc;
}

cudaError_t attn_prepare(int D)
{
    if (D == 64)
        return cudaFuncSetAttribute(frame_attn_lse_importance<64>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    AttnLayout<64>::kAlloc);
    return cudaFuncSetAttribute(frame_attn_lse_importance<128>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                AttnLayout<128>::kAlloc);
}

cudaError_t launch_attn(int D, const CUtensorMap& tm_sk, const CUtensorMap& tm_sv,
                        const CUtensorMap& tm_fk, const CUtensorMap& tm_fv, const AttnParams& p,
                        int U, cudaStream_t st)
{
    const dim3 grid(p.MT, p.Hkv, U);
    if (D == 64)
        frame_attn_lse_importance<64>
            <<<grid, 192, AttnLayout<64>::kAlloc, st>>>(tm_sk, tm_sv, tm_fk, tm_fv, p);
    else
        frame_attn_lse_importance<128>
            <<<grid, 192, AttnLayout<128>::kAlloc, st>>>(tm_sk, tm_sv, tm_fk, tm_fv, p);
    return cudaGetLastError();
}

}  // namespace statekv
