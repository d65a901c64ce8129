// K3: importance reduction, top-B state selection and evict/admit gather
//     (Sec. 3.3, Eq. 6; per layer and KV head as in App. A).
// K4: decode-cache append (Sec. 3.2 detailed state; Sec. 3.3 "append").
//
// K3 runs one CTA per (unit, KV head):
//   1. importance of every pool member = the fixed-order sum of the attention
//      kernel's per-query-tile partials (deterministic); with layer-level
//      selection (App. A) the ranking score is the same sum taken over every
//      KV head of the unit, in one fixed order, so all the unit's CTAs rank
//      identically and their states keep the same positions;
//   2. if the pool (count + T) fits in B, every frame token is admitted;
//      otherwise the B best members by (score desc, position asc) are found
//      with an MSB-first radix select over the 64-bit key
//      (score bits << 32 | ~position) -- scores are non-negative floats, whose
//      bit patterns order like the values, and positions are unique, so the
//      keys are distinct and exactly B members are kept;
//   3. evicted / empty slots (ascending) receive the admitted frame tokens
//      (ascending) as 128-bit row copies, and their positions are updated.
#include "sm103_ptx.cuh"
#include "statekv_kernels.cuh"

#include <algorithm>

namespace statekv {
namespace {

constexpr int kSelThreads = 640;
constexpr int kSelWarps = kSelThreads / 32;
static_assert(kSelWarps <= 32, "one warp combines the warps' values");

// Exclusive block-wide scan of one int per thread; returns the total.
__device__ __forceinline__ int block_exclusive_scan(int x, int* warp_sums, int& excl)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) warp_sums[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        int w = lane < kSelWarps ? warp_sums[lane] : 0;
        int wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += y;
        }
        if (lane < kSelWarps) warp_sums[lane] = wi - w;  // exclusive warp offsets
        if (lane == kSelWarps - 1) warp_sums[kSelWarps] = wi;
    }
    __syncthreads();
    excl = warp_sums[warp] + incl - x;
    return warp_sums[kSelWarps];  // warp_sums is not written again before the caller's next barrier
}

// For each of 8 pool members (columns col[e], active act[e]): the sum of
// x[mt * stride + col] over mt < MT, added in mt order.  Four tiles' loads of
// all 8 members (32 independent loads) are in flight before any addition.
__device__ __forceinline__ void tiles_sum(const float* x, int MT, int stride, const int (&col)[8],
                                          const bool (&act)[8], float (&s)[8])
{
#pragma unroll
    for (int e = 0; e < 8; ++e) s[e] = 0.f;
#pragma unroll 1
    for (int mt = 0; mt < MT; mt += 4) {
        float v[4][8];
#pragma unroll
        for (int m4 = 0; m4 < 4; ++m4)
#pragma unroll
            for (int e = 0; e < 8; ++e)
                v[m4][e] = (act[e] && mt + m4 < MT)
                               ? __ldg(x + static_cast<size_t>(mt + m4) * stride + col[e])
                               : 0.f;
#pragma unroll
        for (int m4 = 0; m4 < 4; ++m4)
#pragma unroll
            for (int e = 0; e < 8; ++e)
                if (mt + m4 < MT) s[e] += v[m4][e];
    }
}

// For 4 adjacent columns c0..c0+3 (16-byte aligned): the sums of
// x[mt * stride + c] over mt < MT, added in mt order, with up to 12 rows'
// 16-byte loads in flight at once (one round of L2 latency for up to 12
// query tiles).
__device__ __forceinline__ float4 rows_sum4(const float* x, int MT, int stride, int c0)
{
    float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 1
    for (int mt = 0; mt < MT; mt += 12) {
        float4 v[12];
#pragma unroll
        for (int m = 0; m < 12; ++m)
            v[m] = mt + m < MT ? __ldg(reinterpret_cast<const float4*>(x + static_cast<size_t>(mt + m) * stride + c0))
                               : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int m = 0; m < 12; ++m)
            if (mt + m < MT) {
                s.x += v[m].x;
                s.y += v[m].y;
                s.z += v[m].z;
                s.w += v[m].w;
            }
    }
    return s;
}

__global__ void __launch_bounds__(kSelThreads)
    state_select_gather(const SelectParams p)
{
    extern __shared__ __align__(16) uint8_t smem_raw[];
    // A kernel launched programmatically behind this one (the transformer
    // block's output projection) may start now: it requests its first weight
    // tiles, which nothing here writes, and waits for this grid's completion
    // before it reads anything else.
    ptx::pdl_launch_dependents();
    const int T = p.T, B = p.B, P = p.P, D = p.D;
    uint64_t* key = reinterpret_cast<uint64_t*>(smem_raw);            // [P]
    int* free_slot = reinterpret_cast<int*>(key + P);                  // [T]
    int* adm_tok = free_slot + T;                                      // [T]
    __shared__ unsigned hist2[2][256];  // pass p counts into hist2[p & 1]; the other is cleared meanwhile
    __shared__ int warp_sums[kSelWarps + 1];
    __shared__ unsigned long long sh_prefix, sh_mask;
    __shared__ int sh_k, sh_done, sh_shift;
    __shared__ unsigned long long warp_and[kSelWarps], warp_or[kSelWarps];

    const int hkv = blockIdx.x, u = blockIdx.y;
    const int ua = p.units.unit_abs(u);
    const int tid = threadIdx.x, lane = tid & 31;
    const size_t head = static_cast<size_t>(ua) * p.Hkv + hkv;
    const int count = p.counts[head];
    const int nf = p.frames[head];
    const int L = nf * T;  // virtual length before this frame
    int32_t* pos = p.positions + head * B;
    const float* part = p.partials + (static_cast<size_t>(u) * p.Hkv + hkv) * p.MT * P;
    float* imp_out =
        p.importance ? p.importance + (static_cast<size_t>(u) * p.Hkv + hkv) * P : nullptr;
    const int n = count + T;
    // the counters come from the arena: a state larger than B or a negative frame
    // count would index past the pool (uniform across the CTA)
    if (!SKV_CHECK(count >= 0 && count <= B && nf >= 0, p.status, 1)) return;

    // 1. importance (fixed-order sum over query tiles) and selection keys.  A
    // thread takes up to 8 pool members at once and walks the query tiles
    // outside them, so all its loads are independent (the partials come from
    // L2); each member's sum still adds the tiles in order.
    const float* part0 = p.partials + static_cast<size_t>(u) * p.Hkv * p.MT * P;
    // bits every selection key shares: the radix select starts below them
    unsigned long long kand = ~0ull, kor = 0ull;
    if ((P & 3) == 0) {
        // Column space, four adjacent columns per thread (16-byte loads): state
        // slot c < count is member c, frame column B + t is member count + t,
        // empty slots are skipped.
        for (int g4 = tid; g4 < (P >> 2); g4 += kSelThreads) {
            const int c0 = 4 * g4;
            int ps[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {  // positions first: their loads overlap the sums'
                // (bounded by B, not by the count, so they do not wait for the count's load)
                const int c = c0 + e;
                ps[e] = c < B ? pos[c] : 0;
            }
            const float4 s4 = rows_sum4(part, p.MT, P, c0);
            float4 r4 = s4;
            if (p.shared) {  // the ranking score: the same sums for every KV head, heads in order
                r4 = make_float4(0.f, 0.f, 0.f, 0.f);
                for (int h2 = 0; h2 < p.Hkv; ++h2) {
                    const float4 t4 = rows_sum4(part0 + static_cast<size_t>(h2) * p.MT * P, p.MT, P, c0);
                    r4.x += t4.x;
                    r4.y += t4.y;
                    r4.z += t4.z;
                    r4.w += t4.w;
                }
            }
            const float sv[4] = {s4.x, s4.y, s4.z, s4.w}, rv[4] = {r4.x, r4.y, r4.z, r4.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int c = c0 + e;
                const int i = c < count ? c : (c >= B && c - B < T) ? count + (c - B) : -1;
                if (i < 0) continue;
                const int pe = c < count ? ps[e] : L + (c - B);
                const uint64_t kk = (static_cast<uint64_t>(__float_as_uint(rv[e])) << 32) |
                                    static_cast<uint32_t>(0xFFFFFFFFu - static_cast<uint32_t>(pe));
                key[i] = kk;
                kand &= kk;
                kor |= kk;
                if (imp_out) imp_out[c] = sv[e];
            }
        }
    } else {  // member-wise: up to 8 pool members per thread
        for (int i0 = 0; i0 < n; i0 += 8 * kSelThreads) {
            int col[8], ps[8];
            bool act[8];
            float s[8], r[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {  // positions first: their loads overlap the sums'
                const int i = i0 + tid + e * kSelThreads;
                act[e] = i < n;
                col[e] = !act[e] ? 0 : i < count ? i : B + (i - count);
                ps[e] = !act[e] ? 0 : i < count ? pos[i] : L + (i - count);
                r[e] = 0.f;
            }
            tiles_sum(part, p.MT, P, col, act, s);
            if (p.shared) {  // the ranking score: the same sums for every KV head, heads in order
                for (int h2 = 0; h2 < p.Hkv; ++h2) {
                    float sh[8];
                    tiles_sum(part0 + static_cast<size_t>(h2) * p.MT * P, p.MT, P, col, act, sh);
#pragma unroll
                    for (int e = 0; e < 8; ++e) r[e] += sh[e];
                }
            }
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                if (!act[e]) continue;
                const int i = i0 + tid + e * kSelThreads;
                const float rank = p.shared ? r[e] : s[e];
                const uint64_t kk = (static_cast<uint64_t>(__float_as_uint(rank)) << 32) |
                                    static_cast<uint32_t>(0xFFFFFFFFu - static_cast<uint32_t>(ps[e]));
                key[i] = kk;
                kand &= kk;
                kor |= kk;
                if (imp_out) imp_out[col[e]] = s[e];
            }
        }
    }
    if (imp_out)
        for (int c = count + tid; c < B; c += kSelThreads) imp_out[c] = 0.f;
    if (B == 0) {  // no compressed state: nothing is kept
        if (tid == 0) p.frames[head] = nf + 1;
        return;
    }

    // 2. top-B selection: kept(i) <=> (key[i] & mask) >= prefix
    unsigned long long prefix = 0, mask = 0;
    if (n > B) {
        {   // block-wide AND and OR of the keys: digits above the highest bit in
            // which two keys differ hold one value for every key, so the radix
            // passes start at the digit holding that bit
            const uint32_t ah = __reduce_and_sync(0xffffffffu, static_cast<uint32_t>(kand >> 32));
            const uint32_t al = __reduce_and_sync(0xffffffffu, static_cast<uint32_t>(kand));
            const uint32_t oh = __reduce_or_sync(0xffffffffu, static_cast<uint32_t>(kor >> 32));
            const uint32_t ol = __reduce_or_sync(0xffffffffu, static_cast<uint32_t>(kor));
            if (lane == 0) {
                warp_and[tid >> 5] = (static_cast<unsigned long long>(ah) << 32) | al;
                warp_or[tid >> 5] = (static_cast<unsigned long long>(oh) << 32) | ol;
            }
        }
        __syncthreads();
        if (tid < 32) {  // warp 0 combines the warps' values
            const unsigned long long wa = lane < kSelWarps ? warp_and[lane] : ~0ull;
            const unsigned long long wo = lane < kSelWarps ? warp_or[lane] : 0ull;
            const unsigned long long a =
                (static_cast<unsigned long long>(__reduce_and_sync(0xffffffffu, static_cast<uint32_t>(wa >> 32)))
                 << 32) |
                __reduce_and_sync(0xffffffffu, static_cast<uint32_t>(wa));
            const unsigned long long o =
                (static_cast<unsigned long long>(__reduce_or_sync(0xffffffffu, static_cast<uint32_t>(wo >> 32)))
                 << 32) |
                __reduce_or_sync(0xffffffffu, static_cast<uint32_t>(wo));
            const unsigned long long diff = a ^ o;  // bits in which some keys differ
            const int hb = diff ? 63 - __clzll(static_cast<long long>(diff)) : 0;
            // the first digit is the 8 bits ending at that bit, so every bit it
            // holds can differ (a digit below bit 0 is cut to its bits >= 0)
            const int shift0 = hb - 7;
            const unsigned long long above = hb >= 63 ? 0ull : ~((2ull << hb) - 1);
            if (lane == 0) {
                sh_shift = shift0;
                sh_prefix = o & above;  // = a & above
                sh_mask = above;
                sh_k = B;
                sh_done = 0;
            }
        }
        for (int i = tid; i < 512; i += kSelThreads) hist2[i >> 8][i & 255] = 0;
        __syncthreads();
        prefix = sh_prefix;
        mask = sh_mask;
        for (int shift = sh_shift, pass = 0; shift > -8; shift -= 8, ++pass) {
            unsigned* hist = hist2[pass & 1];
            const int dsh = shift < 0 ? 0 : shift;                                 // the digit's lowest bit
            const unsigned long long dmask = shift < 0 ? (0xFFull >> -shift) : 0xFFull;  // its bits, at dsh
            for (int i0 = 0; i0 < n; i0 += kSelThreads) {
                const int i = i0 + tid;
                int digit = -1;
                if (i < n && (key[i] & mask) == prefix) digit = static_cast<int>((key[i] >> dsh) & dmask);
                const unsigned peers = __match_any_sync(0xffffffffu, digit);
                if (digit >= 0 && lane == __ffs(peers) - 1) atomicAdd(&hist[digit], __popc(peers));
            }
            __syncthreads();
            if (tid >= 32) {  // the next pass's histogram, while warp 0 reads this one
                for (int i = tid - 32; i < 256; i += kSelThreads - 32) hist2[(pass + 1) & 1][i] = 0;
            } else {
                // lane owns digits 255 - 8*lane - j, j = 0..7 (descending)
                unsigned c[8], local = 0;
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    c[j] = hist[255 - 8 * lane - j];
                    local += c[j];
                }
                unsigned incl = local;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const unsigned y = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += y;
                }
                const unsigned excl = incl - local;
                const int k = sh_k;
                const bool mine = excl < static_cast<unsigned>(k) && incl >= static_cast<unsigned>(k);
                if (mine) {
                    unsigned above = excl;
#pragma unroll 1
                    for (int j = 0; j < 8; ++j) {
                        if (above + c[j] >= static_cast<unsigned>(k)) {
                            const unsigned d = 255 - 8 * lane - j;
                            const int k_rem = k - static_cast<int>(above);
                            sh_prefix = prefix | (static_cast<unsigned long long>(d) << dsh);
                            sh_mask = mask | (dmask << dsh);
                            sh_k = k_rem;
                            sh_done = (c[j] == static_cast<unsigned>(k_rem)) ? 1 : 0;
                            break;
                        }
                        above += c[j];
                    }
                }
            }
            __syncthreads();
            prefix = sh_prefix;
            mask = sh_mask;
            if (sh_done) break;
        }
        __syncthreads();
    } else {
        mask = 0;
        prefix = 0;  // every member kept
    }

    // 3. free slots (evicted or empty, ascending) and admitted tokens (ascending):
    // one block scan over both counts, packed as free + (admitted << 16)
    // (at most kMaxPool < 2^16 free slots, and kMaxFrameTokens admitted)
    const int per = (B + kSelThreads - 1) / kSelThreads;
    const int tper = (T + kSelThreads - 1) / kSelThreads;
    int local_free = 0, local_adm = 0;
    for (int s = tid * per; s < min(B, (tid + 1) * per); ++s)
        local_free += (s >= count || (key[s] & mask) < prefix) ? 1 : 0;
    for (int t = tid * tper; t < min(T, (tid + 1) * tper); ++t)
        local_adm += ((key[count + t] & mask) >= prefix) ? 1 : 0;
    int excl;
    const int tot = block_exclusive_scan(local_free + (local_adm << 16), warp_sums, excl);
    const int nfree = tot & 0xFFFF, nadm = tot >> 16;
    int slot_rank = excl & 0xFFFF, tok_rank = excl >> 16;
    for (int s = tid * per; s < min(B, (tid + 1) * per); ++s)
        if (s >= count || (key[s] & mask) < prefix) {
            if (slot_rank < T) free_slot[slot_rank] = s;
            ++slot_rank;
        }
    for (int t = tid * tper; t < min(T, (tid + 1) * tper); ++t)
        if ((key[count + t] & mask) >= prefix) adm_tok[tok_rank++] = t;
    __syncthreads();
    const int npairs = min(nadm, nfree);
    if (tid == 0 && nadm > nfree) *reinterpret_cast<volatile int32_t*>(p.status) = DEV_BAD_SELECT;

    // 4. gather: 16-byte vector copies of the admitted K and V rows
    const int chunks = D / 8;
    const size_t src_stride = static_cast<size_t>(p.Hkv) * D;
    const __nv_bfloat16* ksrc = p.k + (static_cast<size_t>(u) * T * p.Hkv + hkv) * D;
    const __nv_bfloat16* vsrc = p.v + (static_cast<size_t>(u) * T * p.Hkv + hkv) * D;
    __nv_bfloat16* kdst = p.state_k + head * B * D;
    __nv_bfloat16* vdst = p.state_v + head * B * D;
    for (int w = tid; w < npairs * chunks * 2; w += kSelThreads) {
        const int which = w / (npairs * chunks);
        const int r = w % (npairs * chunks);
        const int i = r / chunks, ch = r % chunks;
        const int t = adm_tok[i], s = free_slot[i];
        if (!SKV_CHECK(t >= 0 && t < T && s >= 0 && s < B, p.status, 2)) continue;
        const __nv_bfloat16* src = (which ? vsrc : ksrc) + t * src_stride + ch * 8;
        __nv_bfloat16* dst = (which ? vdst : kdst) + static_cast<size_t>(s) * D + ch * 8;
        *reinterpret_cast<uint4*>(dst) = *reinterpret_cast<const uint4*>(src);
    }
    for (int i = tid; i < npairs; i += kSelThreads)
        if (SKV_CHECK(free_slot[i] >= 0 && free_slot[i] < B, p.status, 3)) pos[free_slot[i]] = L + adm_tok[i];
    if (tid == 0) {
        p.counts[head] = min(B, count + T);
        p.frames[head] = nf + 1;
    }
}

// K4: D[hkv][L + t][:] = K[t][hkv][:] (and V), one 16-byte chunk per thread.
__global__ void __launch_bounds__(256) decode_cache_append(const AppendParams p)
{
    const int chunks = p.D / 8;
    const long long per_unit = static_cast<long long>(p.T) * p.Hkv * chunks;
    const long long total = 2ll * p.U * per_unit;
    for (long long w = blockIdx.x * 256ll + threadIdx.x; w < total; w += 256ll * gridDim.x) {
        const int which = static_cast<int>(w / (p.U * per_unit));
        const long long r = w % (p.U * per_unit);
        const int u = static_cast<int>(r / per_unit);
        const long long rr = r % per_unit;  // source order [t][hkv][chunk]
        const int t = static_cast<int>(rr / (p.Hkv * chunks));
        const int hkv = static_cast<int>((rr / chunks) % p.Hkv);
        const int ch = static_cast<int>(rr % chunks);
        const int ua = p.units.unit_abs(u);
        const size_t head = static_cast<size_t>(ua) * p.Hkv + hkv;
        const long long row = static_cast<long long>(p.frames[head]) * p.row_mul +
                              (p.row_add ? p.row_add[head] : 0) + t;
        const __nv_bfloat16* src = (which ? p.v : p.k) + static_cast<size_t>(u) * per_unit * 8 +
                                   static_cast<size_t>(rr) * 8;
        __nv_bfloat16* dst = (which ? p.cache_v : p.cache_k) +
                             (head * p.cap + row) * p.D + ch * 8;
        if (!SKV_CHECK(row >= 0 && row < p.cap, p.status, 4)) continue;
        *reinterpret_cast<uint4*>(dst) = *reinterpret_cast<const uint4*>(src);
    }
}

// one CTA of kGuardBytes threads per guard band
__global__ void canary_check(const uint8_t* arena, const GuardList g, int32_t* status)
{
    const int b = blockIdx.x;
    if (b < g.n && arena[g.off[b] + threadIdx.x] != kGuardFill)
        *reinterpret_cast<volatile int32_t*>(status) = DEV_CANARY | (b << 8);
}

}  // namespace

cudaError_t launch_canary_check(const uint8_t* arena, const GuardList& g, int32_t* status, cudaStream_t st)
{
    if (g.n <= 0) return cudaSuccess;
    canary_check<<<g.n, kGuardBytes, 0, st>>>(arena, g, status);
    return cudaGetLastError();
}

size_t select_smem_bytes(int P, int T)
{
    return static_cast<size_t>(P) * 8 + static_cast<size_t>(T) * 8;
}

cudaError_t select_prepare()
{
    return cudaFuncSetAttribute(state_select_gather, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(select_smem_bytes(kMaxPool, kMaxFrameTokens)));
}

cudaError_t launch_select(const SelectParams& p, int U, cudaStream_t st)
{
    const dim3 grid(p.Hkv, U);
    state_select_gather<<<grid, kSelThreads, select_smem_bytes(p.P, p.T), st>>>(p);
    return cudaGetLastError();
}

// Recency window (the baseline the method is compared with): the state keeps
// the B most recent tokens.  Token t of frame n sits at position (n-1) T + t
// and goes to ring slot position mod B, which holds the token B positions
// older -- exactly the one leaving the window -- so no search is needed.
// A flat grid of 16-byte row chunks (like the cache append); a second kernel
// then advances the per-head counters, after every copy has read them.
__global__ void __launch_bounds__(256) state_recency_scatter(const RecencyParams p)
{
    const int t0 = p.T > p.B ? p.T - p.B : 0;  // older frame tokens leave the window at once
    const int nt = p.T - t0, chunks = p.D / 8;
    const long long per_head = static_cast<long long>(nt) * (chunks + 1);  // rows x (chunks + position)
    const long long total = 2ll * p.U * p.Hkv * per_head;
    for (long long w = blockIdx.x * 256ll + threadIdx.x; w < total; w += 256ll * gridDim.x) {
        const int which = static_cast<int>(w / (p.U * p.Hkv * per_head));
        const long long r = w % (p.U * p.Hkv * per_head);
        const int uh = static_cast<int>(r / per_head);
        const int u = uh / p.Hkv, hkv = uh % p.Hkv;
        const long long rr = r % per_head;
        const int t = t0 + static_cast<int>(rr / (chunks + 1));
        const int ch = static_cast<int>(rr % (chunks + 1));
        const size_t head = static_cast<size_t>(p.units.unit_abs(u)) * p.Hkv + hkv;
        const long long pos = static_cast<long long>(p.frames[head]) * p.T + t;
        const long long slot = pos % p.B;
        if (ch == chunks) {  // one thread per row writes its position
            if (which == 0) p.positions[head * p.B + slot] = static_cast<int32_t>(pos);
            continue;
        }
        const __nv_bfloat16* src =
            (which ? p.v : p.k) + ((static_cast<size_t>(u) * p.T + t) * p.Hkv + hkv) * p.D + ch * 8;
        __nv_bfloat16* dst = (which ? p.state_v : p.state_k) + (head * p.B + slot) * p.D + ch * 8;
        *reinterpret_cast<uint4*>(dst) = *reinterpret_cast<const uint4*>(src);
    }
}

__global__ void recency_advance(const RecencyParams p)
{
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= p.U * p.Hkv) return;
    const size_t head = static_cast<size_t>(p.units.unit_abs(i / p.Hkv)) * p.Hkv + i % p.Hkv;
    const long long seen = static_cast<long long>(p.frames[head] + 1) * p.T;
    p.counts[head] = static_cast<int32_t>(seen < p.B ? seen : p.B);
    p.frames[head] += 1;
}

cudaError_t launch_recency(const RecencyParams& p, cudaStream_t st)
{
    if (p.B > 0) {
        const int t0 = p.T > p.B ? p.T - p.B : 0;
        const long long work = 2ll * p.U * p.Hkv * (p.T - t0) * (p.D / 8 + 1);
        const int blocks = static_cast<int>(std::min<long long>((work + 255) / 256, 152ll * 16));
        state_recency_scatter<<<blocks, 256, 0, st>>>(p);
    }
    recency_advance<<<(p.U * p.Hkv + 255) / 256, 256, 0, st>>>(p);
    return cudaGetLastError();
}

__global__ void advance_counter(int32_t* counter, UnitRange units, int U, int Hkv, int n)
{
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= U * Hkv) return;
    counter[static_cast<size_t>(units.unit_abs(i / Hkv)) * Hkv + i % Hkv] += n;
}

cudaError_t launch_advance(int32_t* counter, UnitRange units, int U, int Hkv, int n,
                           cudaStream_t st)
{
    advance_counter<<<(U * Hkv + 255) / 256, 256, 0, st>>>(counter, units, U, Hkv, n);
    return cudaGetLastError();
}

cudaError_t launch_append(const AppendParams& p, cudaStream_t st)
{
    const long long total = 2ll * p.U * p.T * p.Hkv * (p.D / 8);
    const long long blocks = (total + 255) / 256;
    const int grid = static_cast<int>(blocks < 152ll * 64 ? blocks : 152ll * 64);
    decode_cache_append<<<grid, 256, 0, st>>>(p);
    return cudaGetLastError();
}

}  // namespace statekv
