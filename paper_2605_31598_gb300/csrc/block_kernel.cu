// The per-frame transformer block around the StateKV step: the elementwise
// kernels of one decoder layer and the projection GEMMs.
//
//   rmsnorm      y = x / sqrt(mean(x^2) + eps) * g        (fp32, one bf16 rounding)
//   qkv_rope     the QKV projection's q and k rotated at their virtual
//                positions p = L_n + t (Sec. 3.3, "virtual sequence length"),
//                with one fixed RoPE scaling for the whole run ("consistent
//                RoPE scaling"); v copied; written in the step's [T][H][d]
//                layout.  Angles p * theta_k are formed and reduced modulo
//                2 pi in fp64 (p reaches 2^20 and more), then sin/cos in fp32.
//   silu_mul     a = SiLU(gate) * up                       (fp32, one rounding)
//   residual_norm  x += the split-K partials of the output / down projection
//                (summed in split order, one bf16 rounding), then the next
//                RMSNorm of the updated row
//   silu_partials  SiLU * up from the gate/up projection's split-K partials
// The projection GEMMs themselves run on the tensor cores (gemm_kernel.cu).
// Rows are tokens (stream-major, then token): one CTA per row for the norm and
// the rotation, 8 elements per thread for SiLU * up; 16-byte accesses where
// the layout allows.
#include "sm103_ptx.cuh"
#include "statekv_kernels.cuh"

namespace statekv {
namespace {

constexpr int kNormThreads = 512;
constexpr int kNormChunks = 2;  // 8-element chunks a thread keeps: rows up to 8192 wide
constexpr int kSumUnroll = 8;   // split-K partials loaded at once per sum

__device__ __forceinline__ void unpack8(const uint4& u, float (&f)[8])
{
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 t = __bfloat1622float2(h[i]);
        f[2 * i] = t.x;
        f[2 * i + 1] = t.y;
    }
}

__device__ __forceinline__ uint4 pack8(const float (&f)[8])
{
    uint4 u;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
    return u;
}

// The norm of one row held as kNormChunks x 8 floats per thread: sum of
// squares (chunk by chunk, then across the warp and the warps in a fixed
// order), scale 1/sqrt(mean + eps), y = v * scale * g rounded once to bf16.
// Every norm of the block goes through here, so a norm fused into another
// kernel and the standalone one agree bit for bit.
__device__ __forceinline__ void norm_write(const float (&v)[kNormChunks][8], int nc, const uint4* gr,
                                           float eps, int H, uint4* yr, float* red)
{
    float ss = 0.f;
#pragma unroll
    for (int c = 0; c < kNormChunks; ++c) {
        const int i = threadIdx.x + c * kNormThreads;
        if (i < nc)
#pragma unroll
            for (int e = 0; e < 8; ++e) ss += v[c][e] * v[c][e];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < kNormThreads / 32; ++w) tot += red[w];
    const float r = rsqrtf(tot / static_cast<float>(H) + eps);
#pragma unroll
    for (int c = 0; c < kNormChunks; ++c) {
        const int i = threadIdx.x + c * kNormThreads;
        if (i < nc) {
            float gw[8], o[8];
            unpack8(gr[i], gw);
#pragma unroll
            for (int e = 0; e < 8; ++e) o[e] = v[c][e] * r * gw[e];
            yr[i] = pack8(o);
        }
    }
}

// One CTA per row; the row stays in registers between the sum of squares and
// the scaled write (16-byte loads and stores; H a multiple of 8, <= 8192).
__global__ void __launch_bounds__(kNormThreads)
    rmsnorm_kernel(const __nv_bfloat16* x, const __nv_bfloat16* g, float eps, __nv_bfloat16* y,
                   int H)
{
    ptx::pdl_launch_dependents();
    ptx::pdl_wait();
    __shared__ float red[kNormThreads / 32];
    const uint4* xr = reinterpret_cast<const uint4*>(x + static_cast<size_t>(blockIdx.x) * H);
    const int nc = H / 8;
    float v[kNormChunks][8];
#pragma unroll
    for (int c = 0; c < kNormChunks; ++c) {
        const int i = threadIdx.x + c * kNormThreads;
        if (i < nc) unpack8(xr[i], v[c]);
    }
    norm_write(v, nc, reinterpret_cast<const uint4*>(g), eps, H,
               reinterpret_cast<uint4*>(y + static_cast<size_t>(blockIdx.x) * H), red);
}

// One CTA per row: the residual update x += (sum of the split-K partials of
// the projection, in split order), rounded once to bf16, then (when g is set)
// the next RMSNorm of the updated row.
__global__ void __launch_bounds__(kNormThreads)
    residual_norm_kernel(const float* part, int splits, __nv_bfloat16* x, const __nv_bfloat16* g,
                         float eps, __nv_bfloat16* y, int rows, int H)
{
    ptx::pdl_launch_dependents();
    ptx::pdl_wait();
    __shared__ float red[kNormThreads / 32];
    uint4* xr = reinterpret_cast<uint4*>(x + static_cast<size_t>(blockIdx.x) * H);
    const float* pr = part + static_cast<size_t>(blockIdx.x) * H;
    const size_t sstride = static_cast<size_t>(rows) * H;
    const int nc = H / 8;
    float v[kNormChunks][8];
#pragma unroll
    for (int c = 0; c < kNormChunks; ++c) {
        const int i = threadIdx.x + c * kNormThreads;
        if (i < nc) {
            float a[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
            for (int s0 = 0; s0 < splits; s0 += kSumUnroll) {
                float4 lo[kSumUnroll], hi[kSumUnroll];
#pragma unroll
                for (int u = 0; u < kSumUnroll; ++u)
                    if (s0 + u < splits) {
                        const float4* q = reinterpret_cast<const float4*>(pr + (s0 + u) * sstride + 8 * i);
                        lo[u] = __ldcg(q);
                        hi[u] = __ldcg(q + 1);
                    }
#pragma unroll
                for (int u = 0; u < kSumUnroll; ++u)
                    if (s0 + u < splits) {  // split order
                        a[0] += lo[u].x;
                        a[1] += lo[u].y;
                        a[2] += lo[u].z;
                        a[3] += lo[u].w;
                        a[4] += hi[u].x;
                        a[5] += hi[u].y;
                        a[6] += hi[u].z;
                        a[7] += hi[u].w;
                    }
            }
            float xo[8];
            unpack8(xr[i], xo);
#pragma unroll
            for (int e = 0; e < 8; ++e) v[c][e] = __bfloat162float(__float2bfloat16_rn(xo[e] + a[e]));
            xr[i] = pack8(v[c]);
        }
    }
    if (g)
        norm_write(v, nc, reinterpret_cast<const uint4*>(g), eps, H,
                   reinterpret_cast<uint4*>(y + static_cast<size_t>(blockIdx.x) * H), red);
}

// One CTA per token: the d/2 angles of its position are formed once (fp64
// product and reduction modulo 2 pi, fp32 sin/cos) into shared memory, then
// every q and k head's pairs are rotated from that table and v is copied.
__global__ void __launch_bounds__(256) qkv_rope_kernel(const RopeParams p)
{
    ptx::pdl_launch_dependents();
    ptx::pdl_wait();
    __shared__ float cs_tab[64], sn_tab[64];
    const int half = p.d / 2;
    const int row = blockIdx.x;  // s * T + t
    const int s = row / p.T, t = row - s * p.T;
    const __nv_bfloat16* src = p.qkv + static_cast<size_t>(row) * (p.Hq + 2 * p.Hkv) * p.d;
    if (threadIdx.x < half) {
        const long long ua = static_cast<long long>(p.stream_begin + s) * p.num_layers + p.layer;
        const double pos = static_cast<double>(static_cast<long long>(p.frames[ua * p.Hkv]) * p.T + t);
        const double twopi = 6.283185307179586476925286766559;
        double ang = pos * p.freq[threadIdx.x];
        ang -= twopi * floor(ang * (1.0 / twopi));
        float sn, cs;
        sincosf(static_cast<float>(ang), &sn, &cs);
        cs_tab[threadIdx.x] = cs * p.scale;
        sn_tab[threadIdx.x] = sn * p.scale;
    }
    __syncthreads();
    const int qk_pairs = (p.Hq + p.Hkv) * half;
    for (int e = threadIdx.x; e < qk_pairs; e += blockDim.x) {
        const int hh = e / half, k = e - hh * half;
        const float x1 = __bfloat162float(src[hh * p.d + k]);
        const float x2 = __bfloat162float(src[hh * p.d + k + half]);
        const float c = cs_tab[k], sn = sn_tab[k];
        __nv_bfloat16* dst = hh < p.Hq ? p.q + (static_cast<size_t>(row) * p.Hq + hh) * p.d
                                       : p.k + (static_cast<size_t>(row) * p.Hkv + (hh - p.Hq)) * p.d;
        dst[k] = __float2bfloat16(x1 * c - x2 * sn);
        dst[k + half] = __float2bfloat16(x2 * c + x1 * sn);
    }
    const uint4* vs = reinterpret_cast<const uint4*>(src + (p.Hq + p.Hkv) * p.d);
    uint4* vd = reinterpret_cast<uint4*>(p.v + static_cast<size_t>(row) * p.Hkv * p.d);
    for (int e = threadIdx.x; e < p.Hkv * p.d / 8; e += blockDim.x) vd[e] = vs[e];
}

// The same rotation from the QKV projection's split-K partials: CTA
// (row, y) takes 4-column groups [128 y, 128 y + 128) of the row -- a group
// of a q or k head is columns k..k+3 and k+d/2..k+d/2+3 of it, a group of v
// four columns -- and sums each over the splits in split order, adds the
// bias and rounds to bf16 (where the unsplit path stores the projection)
// before rotating.
__device__ __forceinline__ void sum4_splits(const float* col, size_t sstride, int splits, float (&a)[4])
{
    a[0] = a[1] = a[2] = a[3] = 0.f;
    for (int s0 = 0; s0 < splits; s0 += kSumUnroll) {
        float4 f[kSumUnroll];
#pragma unroll
        for (int u = 0; u < kSumUnroll; ++u)
            if (s0 + u < splits) f[u] = __ldcg(reinterpret_cast<const float4*>(col + (s0 + u) * sstride));
#pragma unroll
        for (int u = 0; u < kSumUnroll; ++u)
            if (s0 + u < splits) {
                a[0] += f[u].x;
                a[1] += f[u].y;
                a[2] += f[u].z;
                a[3] += f[u].w;
            }
    }
}

__device__ __forceinline__ void add_bias_round4(const __nv_bfloat16* bias, int col, float (&a)[4])
{
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float b = bias ? __bfloat162float(bias[col + i]) : 0.f;
        a[i] = __bfloat162float(__float2bfloat16_rn(a[i] + b));
    }
}

__device__ __forceinline__ uint2 pack4(float a, float b, float c, float d)
{
    return make_uint2(ptx::pack_bf16x2(a, b), ptx::pack_bf16x2(c, d));
}

constexpr int kRopeGroups = 128;  // 4-column groups (threads) per CTA

__global__ void __launch_bounds__(kRopeGroups) qkv_rope_partials_kernel(const RopeParams p)
{
    ptx::pdl_launch_dependents();
    ptx::pdl_wait();
    __shared__ float cs_tab[64], sn_tab[64];
    const int half = p.d / 2, hg = half / 4;  // groups per rotated head
    const int row = blockIdx.x;               // s * T + t
    const int s = row / p.T, t = row - s * p.T;
    if (threadIdx.x < half) {
        const long long ua = static_cast<long long>(p.stream_begin + s) * p.num_layers + p.layer;
        const double pos = static_cast<double>(static_cast<long long>(p.frames[ua * p.Hkv]) * p.T + t);
        const double twopi = 6.283185307179586476925286766559;
        double ang = pos * p.freq[threadIdx.x];
        ang -= twopi * floor(ang * (1.0 / twopi));
        float sn, cs;
        sincosf(static_cast<float>(ang), &sn, &cs);
        cs_tab[threadIdx.x] = cs * p.scale;
        sn_tab[threadIdx.x] = sn * p.scale;
    }
    __syncthreads();
    const int width = (p.Hq + 2 * p.Hkv) * p.d;
    const size_t sstride = static_cast<size_t>(p.S) * p.T * width;
    const float* prow = p.part + static_cast<size_t>(row) * width;
    const int g = blockIdx.y * kRopeGroups + threadIdx.x;
    const int qk_groups = (p.Hq + p.Hkv) * hg;
    if (g < qk_groups) {
        const int hh = g / hg, k = 4 * (g - hh * hg);
        const int c1 = hh * p.d + k, c2 = c1 + half;
        float x1[4], x2[4];
        sum4_splits(prow + c1, sstride, p.splits, x1);
        sum4_splits(prow + c2, sstride, p.splits, x2);
        add_bias_round4(p.bias, c1, x1);
        add_bias_round4(p.bias, c2, x2);
        float o1[4], o2[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float c = cs_tab[k + i], sn = sn_tab[k + i];
            o1[i] = x1[i] * c - x2[i] * sn;
            o2[i] = x2[i] * c + x1[i] * sn;
        }
        __nv_bfloat16* dst = hh < p.Hq ? p.q + (static_cast<size_t>(row) * p.Hq + hh) * p.d
                                       : p.k + (static_cast<size_t>(row) * p.Hkv + (hh - p.Hq)) * p.d;
        *reinterpret_cast<uint2*>(dst + k) = pack4(o1[0], o1[1], o1[2], o1[3]);
        *reinterpret_cast<uint2*>(dst + k + half) = pack4(o2[0], o2[1], o2[2], o2[3]);
    } else if (g < qk_groups + p.Hkv * p.d / 4) {
        const int e = 4 * (g - qk_groups);
        const int c = (p.Hq + p.Hkv) * p.d + e;
        float x[4];
        sum4_splits(prow + c, sstride, p.splits, x);
        add_bias_round4(p.bias, c, x);
        *reinterpret_cast<uint2*>(p.v + static_cast<size_t>(row) * p.Hkv * p.d + e) = pack4(x[0], x[1], x[2], x[3]);
    }
}

// 8 outputs per thread: a = SiLU(gate) * up, gate in columns [0, I), up in [I, 2I).
__global__ void silu_mul_kernel(const __nv_bfloat16* gu, __nv_bfloat16* a, int rows, int I)
{
    ptx::pdl_launch_dependents();
    ptx::pdl_wait();
    const int chunks = I / 8;
    const long long idx = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= static_cast<long long>(rows) * chunks) return;
    const int r = static_cast<int>(idx / chunks), c = static_cast<int>(idx - static_cast<long long>(r) * chunks);
    const uint4* grow = reinterpret_cast<const uint4*>(gu + static_cast<size_t>(r) * 2 * I);
    float g[8], u[8], o[8];
    unpack8(grow[c], g);
    unpack8(grow[chunks + c], u);
#pragma unroll
    for (int e = 0; e < 8; ++e) o[e] = g[e] / (1.f + expf(-g[e])) * u[e];
    reinterpret_cast<uint4*>(a + static_cast<size_t>(r) * I)[c] = pack8(o);
}

// 8 outputs per thread from split-K partials: gate and up summed in split
// order and rounded to bf16 (where the unsplit path stores them), then
// a = SiLU(gate) * up.
__global__ void silu_partials_kernel(const float* part, int splits, __nv_bfloat16* a, int rows, int I)
{
    ptx::pdl_launch_dependents();
    ptx::pdl_wait();
    const int chunks = I / 8;
    const long long idx = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= static_cast<long long>(rows) * chunks) return;
    const int r = static_cast<int>(idx / chunks), c = static_cast<int>(idx - static_cast<long long>(r) * chunks);
    const float* pr = part + static_cast<size_t>(r) * 2 * I + 8 * c;
    const size_t sstride = static_cast<size_t>(rows) * 2 * I;
    float g[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f}, u[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll 2
    for (int sp = 0; sp < splits; ++sp) {
        const float4* qg = reinterpret_cast<const float4*>(pr + sp * sstride);
        const float4* qu = reinterpret_cast<const float4*>(pr + sp * sstride + I);
        const float4 g0 = __ldcg(qg), g1 = __ldcg(qg + 1), u0 = __ldcg(qu), u1 = __ldcg(qu + 1);
        g[0] += g0.x; g[1] += g0.y; g[2] += g0.z; g[3] += g0.w;
        g[4] += g1.x; g[5] += g1.y; g[6] += g1.z; g[7] += g1.w;
        u[0] += u0.x; u[1] += u0.y; u[2] += u0.z; u[3] += u0.w;
        u[4] += u1.x; u[5] += u1.y; u[6] += u1.z; u[7] += u1.w;
    }
    float o[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const float gb = __bfloat162float(__float2bfloat16_rn(g[e]));
        const float ub = __bfloat162float(__float2bfloat16_rn(u[e]));
        o[e] = gb / (1.f + expf(-gb)) * ub;
    }
    reinterpret_cast<uint4*>(a + static_cast<size_t>(r) * I)[c] = pack8(o);
}

// Every kernel of the block is launched with programmatic stream
// serialization: it starts launching while the previous kernel finishes and
// waits (pdl_wait, first thing) for that kernel's completion before it reads
// or writes anything.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, cudaStream_t st, Args... args)
{
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = 0;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

}  // namespace

cudaError_t launch_residual_norm(const float* part, int splits, __nv_bfloat16* x,
                                 const __nv_bfloat16* g, float eps, __nv_bfloat16* y, int rows,
                                 int H, cudaStream_t st)
{
    if (rows <= 0) return cudaSuccess;
    return launch_pdl(residual_norm_kernel, dim3(rows), dim3(kNormThreads), st, part, splits, x, g, eps, y,
                      rows, H);
}

cudaError_t launch_silu_partials(const float* part, int splits, __nv_bfloat16* a, int rows, int I,
                                 cudaStream_t st)
{
    const long long total = static_cast<long long>(rows) * (I / 8);
    if (total <= 0) return cudaSuccess;
    return launch_pdl(silu_partials_kernel, dim3(static_cast<unsigned>((total + 255) / 256)), dim3(256), st,
                      part, splits, a, rows, I);
}

cudaError_t launch_rmsnorm(const __nv_bfloat16* x, const __nv_bfloat16* g, float eps,
                           __nv_bfloat16* y, int rows, int H, cudaStream_t st)
{
    if (rows <= 0) return cudaSuccess;
    return launch_pdl(rmsnorm_kernel, dim3(rows), dim3(kNormThreads), st, x, g, eps, y, H);
}

cudaError_t launch_qkv_rope(const RopeParams& p, cudaStream_t st)
{
    const int rows = p.S * p.T;
    if (rows <= 0) return cudaSuccess;
    if (p.part) {
        const int groups = (p.Hq + p.Hkv) * (p.d / 8) + p.Hkv * p.d / 4;
        return launch_pdl(qkv_rope_partials_kernel, dim3(rows, (groups + kRopeGroups - 1) / kRopeGroups),
                          dim3(kRopeGroups), st, p);
    }
    return launch_pdl(qkv_rope_kernel, dim3(rows), dim3(256), st, p);
}

cudaError_t launch_silu_mul(const __nv_bfloat16* gu, __nv_bfloat16* a, long long rows, int I,
                            cudaStream_t st)
{
    const long long total = rows * (I / 8);
    if (total <= 0) return cudaSuccess;
    return launch_pdl(silu_mul_kernel, dim3(static_cast<unsigned>((total + 255) / 256)), dim3(256), st, gu, a,
                      static_cast<int>(rows), I);
}

}  // namespace statekv
