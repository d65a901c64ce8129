// App. A assumption diagnostics on the GPU.
//
//   scores_reduce       layer-level score of every key of a full-attention
//                       frame: the attention kernel's per-(KV head, query
//                       tile) partials summed in one fixed order (App. A's
//                       shared protocol sums the weights over the frame's
//                       queries within each head, then over the heads)
//   topb_mask           top-B membership of each row, ties to the lower
//                       position: an MSB-first radix select over the 64-bit
//                       key (score bits << 32 | ~position), read from global
//                       memory on every pass, so rows may be arbitrarily long
//   concentration_sums  App. A.1: mass of the top-B historical keys and of
//                       all historical keys
//   state_metrics       App. A.2: the counts and weights behind candidate-pool
//                       recall, weighted recall, retention and churn
// Every reduction is one CTA per row with a fixed-order fp64 tree, so the
// results are deterministic.
#include "statekv_kernels.cuh"

namespace statekv {
namespace {

constexpr int kDiagThreads = 512;

// Sum of one double per thread over the block; thread 0 gets the total.
__device__ double block_sum(double x, double* sh)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_down_sync(0xffffffffu, x, o);
    if (lane == 0) sh[warp] = x;
    __syncthreads();
    double t = 0.0;
    if (warp == 0) {
        t = lane < kDiagThreads / 32 ? sh[lane] : 0.0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) t += __shfl_down_sync(0xffffffffu, t, o);
    }
    __syncthreads();
    return t;
}

__global__ void scores_reduce(const ScoresParams p)
{
    const int u = blockIdx.y;
    const long long j = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (j >= p.ncols) return;
    const int ua = p.units.unit_abs(u);
    const long long L = static_cast<long long>(p.frames[static_cast<size_t>(ua) * p.Hkv]) * p.T;
    float s = 0.f;
    if (j < L + p.T) {
        const long long col = j < L ? j : p.Bp + (j - L);
        const float* part = p.partials + static_cast<size_t>(u) * p.Hkv * p.MT * p.Pp + col;
        for (int h = 0; h < p.Hkv; ++h) {
            float sh = 0.f;  // one KV head: its query tiles in order
            for (int mt = 0; mt < p.MT; ++mt)
                sh += part[(static_cast<size_t>(h) * p.MT + mt) * p.Pp];
            s += sh;
        }
    }
    p.scores[static_cast<size_t>(u) * p.ncols + j] = s;
}

// Selection key of entry j: order-preserving bits of the (non-negative)
// score, then the complement of the position so that the lower position wins
// a tie.  Negative scores and NaN count as 0.
__device__ __forceinline__ unsigned long long topb_key(const float* row, long long j)
{
    const float x = row[j];
    const float c = x > 0.f ? x : 0.f;  // also maps NaN to 0
    return (static_cast<unsigned long long>(__float_as_uint(c)) << 32) |
           static_cast<unsigned>(0xFFFFFFFFu - static_cast<unsigned>(j));
}

__global__ void __launch_bounds__(kDiagThreads) topb_mask_kernel(const float* scores, long long n,
                                                                 long long stride, long long B,
                                                                 uint8_t* mask)
{
    __shared__ unsigned hist[256];
    __shared__ unsigned long long sh_prefix, sh_mask;
    __shared__ long long sh_k;
    __shared__ int sh_done;
    const float* row = scores + static_cast<size_t>(blockIdx.x) * stride;
    uint8_t* mrow = mask + static_cast<size_t>(blockIdx.x) * stride;
    const int tid = threadIdx.x, lane = tid & 31;
    unsigned long long prefix = 0, msk = 0;
    bool none = B <= 0;
    if (!none && n > B) {
        if (tid == 0) {
            sh_k = B;
            sh_done = 0;
        }
        __syncthreads();
        for (int shift = 56; shift >= 0; shift -= 8) {
            for (int i = tid; i < 256; i += kDiagThreads) hist[i] = 0;
            __syncthreads();
            for (long long i0 = 0; i0 < n; i0 += kDiagThreads) {
                const long long i = i0 + tid;
                int digit = -1;
                if (i < n) {
                    const unsigned long long k = topb_key(row, i);
                    if ((k & msk) == prefix) digit = static_cast<int>((k >> shift) & 0xFF);
                }
                const unsigned peers = __match_any_sync(0xffffffffu, digit);
                if (digit >= 0 && lane == __ffs(peers) - 1) atomicAdd(&hist[digit], __popc(peers));
            }
            __syncthreads();
            if (tid < 32) {
                // lane owns digits 255 - 8 lane - e, e = 0..7 (descending)
                unsigned c[8], local = 0;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    c[e] = hist[255 - 8 * lane - e];
                    local += c[e];
                }
                unsigned incl = local;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const unsigned y = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += y;
                }
                const unsigned long long excl = incl - local;
                const long long k = sh_k;
                if (static_cast<long long>(excl) < k && static_cast<long long>(incl) >= k) {
                    long long above = static_cast<long long>(excl);
#pragma unroll 1
                    for (int e = 0; e < 8; ++e) {
                        if (above + c[e] >= k) {
                            const unsigned long long dgt = 255 - 8 * lane - e;
                            sh_prefix = prefix | (dgt << shift);
                            sh_mask = msk | (0xFFull << shift);
                            sh_k = k - above;
                            sh_done = (static_cast<long long>(c[e]) == k - above) ? 1 : 0;
                            break;
                        }
                        above += c[e];
                    }
                }
            }
            __syncthreads();
            prefix = sh_prefix;
            msk = sh_mask;
            if (sh_done) break;
        }
    }
    // kept(j) <=> j < n and (key(j) & mask) >= prefix (prefix 0: every entry)
    for (long long j = tid; j < stride; j += kDiagThreads) {
        uint8_t keep = 0;
        if (!none && j < n) keep = (topb_key(row, j) & msk) >= prefix ? 1 : 0;
        mrow[j] = keep;
    }
}

__global__ void __launch_bounds__(kDiagThreads) concentration_kernel(const float* scores,
                                                                     const uint8_t* mask,
                                                                     long long n, long long stride,
                                                                     double* out)
{
    __shared__ double sh[kDiagThreads / 32];
    const float* row = scores + static_cast<size_t>(blockIdx.x) * stride;
    const uint8_t* mrow = mask + static_cast<size_t>(blockIdx.x) * stride;
    double top = 0.0, all = 0.0;
    for (long long j = threadIdx.x; j < n; j += kDiagThreads) {
        const double x = row[j];
        all += x;
        if (mrow[j]) top += x;
    }
    top = block_sum(top, sh);
    all = block_sum(all, sh);
    if (threadIdx.x == 0) {
        out[2 * blockIdx.x] = top;
        out[2 * blockIdx.x + 1] = all;
    }
}

__global__ void __launch_bounds__(kDiagThreads) state_metrics_kernel(
    const uint8_t* mask_n, const uint8_t* mask_n1, const float* w, long long n_seen, int T,
    long long stride, double* out)
{
    __shared__ double sh[kDiagThreads / 32];
    const size_t base = static_cast<size_t>(blockIdx.x) * stride;
    double v[6] = {0.0, 0.0, 0.0, 0.0, 0.0, 0.0};
    for (long long j = threadIdx.x; j < n_seen + T; j += kDiagThreads) {
        const bool in_n = j < n_seen && mask_n[base + j];
        const bool in_n1 = mask_n1[base + j] != 0;
        const bool in_pool = in_n || j >= n_seen;  // S_n plus frame n + 1
        const double x = w[base + j];
        if (in_n1) {
            v[1] += 1.0;
            v[3] += x;
            if (in_pool) {
                v[0] += 1.0;
                v[2] += x;
            }
            if (in_n) v[4] += 1.0;
        }
        if (in_n) v[5] += 1.0;
    }
#pragma unroll 1
    for (int i = 0; i < 6; ++i) {
        const double t = block_sum(v[i], sh);
        if (threadIdx.x == 0) out[6 * blockIdx.x + i] = t;
    }
}

}  // namespace

cudaError_t launch_scores_reduce(const ScoresParams& p, int U, cudaStream_t st)
{
    if (U <= 0 || p.ncols <= 0) return cudaSuccess;
    const dim3 grid(static_cast<unsigned>((p.ncols + 255) / 256), static_cast<unsigned>(U));
    scores_reduce<<<grid, 256, 0, st>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_topb_mask(const float* scores, int rows, long long n, long long stride,
                             long long B, uint8_t* mask, cudaStream_t st)
{
    if (rows <= 0) return cudaSuccess;
    topb_mask_kernel<<<rows, kDiagThreads, 0, st>>>(scores, n, stride, B, mask);
    return cudaGetLastError();
}

cudaError_t launch_concentration(const float* scores, const uint8_t* mask, int rows, long long n,
                                 long long stride, double* out, cudaStream_t st)
{
    if (rows <= 0) return cudaSuccess;
    concentration_kernel<<<rows, kDiagThreads, 0, st>>>(scores, mask, n, stride, out);
    return cudaGetLastError();
}

cudaError_t launch_state_metrics(const uint8_t* mask_n, const uint8_t* mask_n1, const float* w,
                                 int rows, long long n_seen, int T, long long stride, double* out,
                                 cudaStream_t st)
{
    if (rows <= 0) return cudaSuccess;
    state_metrics_kernel<<<rows, kDiagThreads, 0, st>>>(mask_n, mask_n1, w, n_seen, T, stride, out);
    return cudaGetLastError();
}

}  // namespace statekv
