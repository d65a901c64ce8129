// The per-frame transformer block around the StateKV step: the elementwise
// kernels of one decoder layer and the projection GEMMs.
//
//   rmsnorm      y = x / sqrt(mean(x^2) + eps) * g        (fp32, one bf16 rounding);
//                optionally also the cos/sin table of the rows' virtual
//                positions for the next QKV projection's epilogue
//   qkv_rope     the QKV projection's q and k rotated at their virtual
//                positions p = L_n + t (Sec. 3.3, "virtual sequence length"),
//                with one fixed RoPE scaling for the whole run ("consistent
//                RoPE scaling"); v copied; written in the step's [T][H][d]
//                layout.  Angles p * theta_k are formed and reduced modulo
//                2 pi in fp64 (p reaches 2^20 and more), then sin/cos in fp32.
//   silu_mul     a = SiLU(gate) * up                       (fp32, one rounding)
// The projection GEMMs themselves run on the tensor cores (gemm_kernel.cu);
// up to 256 rows their epilogues also do the bias, the rotation, the residual
// update and SiLU * up.  Rows are tokens (stream-major, then token): one CTA
// per row for the norm and the rotation, 8 elements per thread for SiLU * up;
// 16-byte accesses where the layout allows.
#include "sm103_ptx.cuh"
#include "statekv_kernels.cuh"

namespace statekv {
namespace {

constexpr int kNormThreads = 512;
constexpr int kNormChunks = 2;  // 8-element chunks a thread keeps: rows up to 8192 wide

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

// The angles of one row's virtual position: fp64 product and reduction
// modulo 2 pi, fp32 sin/cos, the RoPE scaling's factor applied.
__device__ __forceinline__ float2 rope_angle(const RopeParams& p, int row, int k)
{
    const int s = row / p.T, t = row - s * p.T;
    const long long ua = static_cast<long long>(p.stream_begin + s) * p.num_layers + p.layer;
    const double pos = static_cast<double>(static_cast<long long>(p.frames[ua * p.Hkv]) * p.T + t);
    const double twopi = 6.283185307179586476925286766559;
    double ang = pos * p.freq[k];
    ang -= twopi * floor(ang * (1.0 / twopi));
    float sn, cs;
    sincosf(static_cast<float>(ang), &sn, &cs);
    return make_float2(cs * p.scale, sn * p.scale);
}

// One CTA per row; the row stays in registers between the sum of squares and
// the scaled write (16-byte loads and stores; H a multiple of 8, <= 8192).
// With `rope` set, threads [0, d/2) also write the row's (cos, sin) table
// (rp.d <= 128, so d/2 <= kNormThreads).
__global__ void __launch_bounds__(kNormThreads)
    rmsnorm_kernel(const __nv_bfloat16* x, const __nv_bfloat16* g, float eps, __nv_bfloat16* y,
                   int H, const RopeParams rp, float2* rope)
{
    ptx::pdl_launch_dependents();
    ptx::pdl_wait();
    if (rope && threadIdx.x < rp.d / 2)
        rope[static_cast<size_t>(blockIdx.x) * (rp.d / 2) + threadIdx.x] = rope_angle(rp, blockIdx.x, threadIdx.x);
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
    const __nv_bfloat16* src = p.qkv + static_cast<size_t>(row) * (p.Hq + 2 * p.Hkv) * p.d;
    if (threadIdx.x < half) {
        const float2 a = rope_angle(p, row, threadIdx.x);
        cs_tab[threadIdx.x] = a.x;
        sn_tab[threadIdx.x] = a.y;
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

cudaError_t launch_rmsnorm(const __nv_bfloat16* x, const __nv_bfloat16* g, float eps,
                           __nv_bfloat16* y, int rows, int H, cudaStream_t st)
{
    if (rows <= 0) return cudaSuccess;
    return launch_pdl(rmsnorm_kernel, dim3(rows), dim3(kNormThreads), st, x, g, eps, y, H, RopeParams{},
                      static_cast<float2*>(nullptr));
}

cudaError_t launch_rmsnorm_rope(const __nv_bfloat16* x, const __nv_bfloat16* g, float eps,
                                __nv_bfloat16* y, int rows, int H, const RopeParams& rp, float2* rope,
                                cudaStream_t st)
{
    if (rows <= 0) return cudaSuccess;
    if (!rope || rp.d < 2 || rp.d > 128 || rows != rp.S * rp.T) return cudaErrorInvalidValue;
    return launch_pdl(rmsnorm_kernel, dim3(rows), dim3(kNormThreads), st, x, g, eps, y, H, rp, rope);
}

cudaError_t launch_qkv_rope(const RopeParams& p, cudaStream_t st)
{
    const int rows = p.S * p.T;
    if (rows <= 0) return cudaSuccess;
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
