// Kernel parameter blocks and launchers of the StateKV per-frame step.
//
//   K4  decode-cache append   (Sec. 3.2 / 3.3: D_n = D_{n-1} + (K_n, V_n))
//   K1  frame attention + LSE + fused importance partials (Eq. 5, Eq. 1, App. B.1)
//   K3  importance reduction, top-B select, evict/admit gather (Eq. 6)
//
// A "unit" is one (stream, layer) of the current call; `unit_abs` indexes the
// arena (stream * num_layers + layer), `u` indexes the call's buffers.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

namespace statekv {

// Device error codes written to the status word (0 = no error).  The low
// byte is the kind; an attention-kernel timeout carries the waiting site in
// bits 8..15 (the first expired wait of the CTA): 1 the watchdog self-test's
// barrier (see AttnParams::selftest_stall), 2 producer (free slot),
// 4..9 MMA issuer X (4 Q ready, 5 K tile landed, 6 score buffer free, 7 P
// written, 8 V tile landed, 9 pass A done and read; +16 for issuer Y),
// 10..12 and 14 softmax warpgroup 0 (10 Q K^T in pass A, 11 pass-B scores
// ready, 12 the P buffer or the staging area free, 14 O final; +32 for
// warpgroup 1), 13 the column-sum reducer.
enum DeviceError : int32_t {
    DEV_OK = 0,
    DEV_TIMEOUT_ATTN = 1,
    DEV_BAD_SELECT = 2,  // the top-B selection admitted more tokens than free slots
    DEV_TIMEOUT_GEMM = 3,  // a projection-GEMM wait expired (bits 8..15: 2 producer,
                           // 3 MMA issuer stage, 4 MMA issuer accumulator, 5 epilogue)
    DEV_TIMEOUT_DECODE = 4,  // a decode kernel's wait for its K/V copies expired
    DEV_BOUNDS = 5,          // debug builds: an index failed its bounds check (bits 8..15: site)
    DEV_CANARY = 6,          // debug builds: an arena guard band was overwritten (bits 8..15: band)
};

// Debug builds (STATEKV_DEBUG_CHECKS=1) check indices before the accesses
// marked with SKV_CHECK: a failed check records DEV_BOUNDS with its site in
// the status word (unless a failure is already recorded) and the access is
// skipped; no trap.
// Release builds compile every check to `true`.
#ifndef STATEKV_DEBUG_CHECKS
#define STATEKV_DEBUG_CHECKS 0
#endif
#if STATEKV_DEBUG_CHECKS
__device__ __forceinline__ bool skv_check(bool ok, int32_t* status, int site)
{
    // the status word may live in mapped host memory: a plain store, no atomic
    if (!ok && status && *reinterpret_cast<volatile int32_t*>(status) == 0)
        *reinterpret_cast<volatile int32_t*>(status) = DEV_BOUNDS | (site << 8);
    return ok;
}
#define SKV_CHECK(cond, status, site) (::statekv::skv_check((cond), (status), (site)))
#else
#define SKV_CHECK(cond, status, site) true
#endif

// Tile sizes of the attention kernel: 128 query rows x 128 keys per MMA tile.
constexpr int kBM = 128;
constexpr int kBN = 128;

struct UnitRange {
    int stream_begin, layer_begin, layer_count, num_layers;
    __host__ __device__ int unit_abs(int u) const
    {
        return (stream_begin + u / layer_count) * num_layers + layer_begin + u % layer_count;
    }
};

struct AttnParams {
    const __nv_bfloat16* q;   // [U][T][Hq][D]
    __nv_bfloat16* out;       // [U][T][Hq][D]
    float* partials;          // [U][Hkv][MT][P]; null: no importance (full attention)
    const int32_t* counts;    // arena [S*L][Hkv]: visible keys before the frame =
                              //   counts * count_mul + (count_add ? count_add : 0)
    const int32_t* count_add; // nullable arena [S*L][Hkv]
    int32_t* status;          // device-visible status word
    UnitRange units;
    int T, Hq, Hkv, G, B, P, MT;
    int U;                    // units of the call (set by launch_attn)
    int causal;
    int count_mul;            // 1: counts are state sizes; T: counts are frame counters
    float scale_log2;         // softmax scale * log2(e)
    unsigned long long watchdog_ns;
    // Watchdog self-test: 1 makes the producer wait first on a barrier that
    // nothing completes, so its bounded wait expires and the CTA aborts
    // through the regular timeout path (no copy or MMA is issued).
    int selftest_stall;
};

struct SelectParams {
    const float* partials;      // [U][Hkv][MT][P]
    float* importance;          // nullable [U][Hkv][P]
    const __nv_bfloat16* k;     // [U][T][Hkv][D]
    const __nv_bfloat16* v;
    __nv_bfloat16* state_k;     // arena [S*L][Hkv][B][D]
    __nv_bfloat16* state_v;
    int32_t* positions;         // arena [S*L][Hkv][B]
    int32_t* counts;            // arena [S*L][Hkv]
    int32_t* frames;            // arena [S*L][Hkv]
    int32_t* status;
    UnitRange units;
    int T, Hkv, D, B, P, MT;
    int shared;                 // 1: rank by the importance summed over every KV head
};

struct AppendParams {
    const __nv_bfloat16* k;     // [U][T][Hkv][D]: T rows per unit appended
    const __nv_bfloat16* v;
    __nv_bfloat16* cache_k;     // arena [S*L][Hkv][cap][D]
    __nv_bfloat16* cache_v;
    const int32_t* frames;      // arena [S*L][Hkv]
    const int32_t* row_add;     // nullable arena [S*L][Hkv]: rows already past frames * row_mul
    UnitRange units;
    int U, T, Hkv, D;
    int row_mul;                // first row = frames * row_mul + row_add
    long long cap;
    int32_t* status;            // debug builds: bounds-check failures
};

struct RecencyParams {
    const __nv_bfloat16* k;     // [U][T][Hkv][D]
    const __nv_bfloat16* v;
    __nv_bfloat16* state_k;     // arena [S*L][Hkv][B][D], slot = position mod B
    __nv_bfloat16* state_v;
    int32_t* positions;         // arena [S*L][Hkv][B]
    int32_t* counts;            // arena [S*L][Hkv]
    int32_t* frames;            // arena [S*L][Hkv]
    UnitRange units;
    int U, T, Hkv, D, B;
};

struct ScoresParams {
    const float* partials;      // [U][Hkv][MT][Pp] from the attention kernel
    float* scores;              // [U][ncols]
    const int32_t* frames;      // arena [S*L][Hkv]: frames before this one
    UnitRange units;
    int T, Hkv, MT;
    long long Bp, Pp;           // frame keys sit at partial columns Bp + t; Pp = Bp + T
    long long ncols;            // row length of scores (>= keys of every unit)
};

// App. A diagnostics (diag_kernel.cu).
cudaError_t launch_scores_reduce(const ScoresParams& p, int U, cudaStream_t st);
cudaError_t launch_topb_mask(const float* scores, int rows, long long n, long long stride,
                             long long B, uint8_t* mask, cudaStream_t st);
cudaError_t launch_concentration(const float* scores, const uint8_t* mask, int rows, long long n,
                                 long long stride, double* out, cudaStream_t st);
cudaError_t launch_state_metrics(const uint8_t* mask_n, const uint8_t* mask_n1, const float* w,
                                 int rows, long long n_seen, int T, long long stride, double* out,
                                 cudaStream_t st);

// Per-frame transformer block (block_kernel.cu).
struct RopeParams {
    const __nv_bfloat16* qkv;   // [S*T][(Hq + 2 Hkv) * d]: q heads, k heads, v heads
    __nv_bfloat16* q;           // [S][T][Hq][d]
    __nv_bfloat16* k;           // [S][T][Hkv][d]
    __nv_bfloat16* v;           // [S][T][Hkv][d]
    const int32_t* frames;      // arena [S*L][Hkv]: frames before this one
    int stream_begin, layer, num_layers;
    int S, T, Hq, Hkv, d;
    float scale;                // q and k scale of the RoPE scaling (1: none)
    double freq[64];            // angular frequency of rotated pair k < d / 2
};
cudaError_t launch_rmsnorm(const __nv_bfloat16* x, const __nv_bfloat16* g, float eps,
                           __nv_bfloat16* y, int rows, int H, cudaStream_t st);
cudaError_t launch_qkv_rope(const RopeParams& p, cudaStream_t st);
cudaError_t launch_silu_mul(const __nv_bfloat16* gu, __nv_bfloat16* a, long long rows, int I,
                            cudaStream_t st);
// Projection GEMMs of the block (gemm_kernel.cu): D[M][N] = X[M][K] W[N][K]^T
// (+ bias[N]) (+ D when add), bf16, fp32 accumulation on tcgen05.  A unit is
// a 128-column tile of W for a pair of 128-row tiles of X over kps 64-wide K
// steps; splits > 1 writes fp32 partials [units][2][128][128] and, in a
// cooperative launch, every split of a tile waits for its siblings
// (counters[tile], zero on entry, left at `splits`) and adds its share of the
// tile's rows over all splits in split order.
constexpr int kGemmBM = 128, kGemmBN = 128, kGemmBK = 64;
struct GemmPlan {
    int bn;                     // W rows per tile: 128, or 192 / 256 for GEMMs with many tiles (no K split)
    int n_tiles, m_pairs, k_steps, kps, splits, units, counters;
    size_t partial_bytes;
};
GemmPlan gemm_plan(int M, int N, int K, int sms);
struct GemmParams {
    int M, N, K;
    int bn;                     // the plan's tile width; the W tensor map's box has bn rows
    int n_tiles, k_steps, kps, splits, units;
    int paired_I;               // > 0: W = gate rows [0, I) then up rows [I, 2 I), D = SiLU(gate) * up
                                // [M][I] (N = I); the W map is [2][I][K] with boxes of bn / 2 rows,
                                // tile t covers output columns [t bn / 2, (t + 1) bn / 2); splits = 1
    const __nv_bfloat16* bias;  // nullable [N]
    __nv_bfloat16* D;           // [M][N]
    int add;                    // 1: D += X W^T
    float* partials;            // splits > 1: [units][2][128][128]
    int* counters;              // splits > 1: [n_tiles * m_pairs], zero on entry, used once
    int32_t* status;
    unsigned long long watchdog_ns;
};
cudaError_t gemm_prepare();
cudaError_t launch_gemm(const CUtensorMap& tm_x, const CUtensorMap& tm_w, const GemmParams& p,
                        int sms, cudaStream_t st);
// Thin projections (M <= kThinMaxRows rows, gemm_kernel.cu): W is the MMA's
// A operand and all of X (Mp = M rounded up to 16 rows, one TMA box of 64
// K-columns x Mp rows) its B operand.  A unit is `wblocks` 128-row blocks of
// W (rows [256 t, 256 t + 256) for two; for the gate/up projection a gate
// block and the matching up block) over one range of K; the `splits` units of
// a tile form a thread-block cluster, which adds its accumulators in
// distributed shared memory in rank order, each CTA finishing a 1/splits
// share of the rows of X:
//   kThinResidual  out[m][n] = bf16(out[m][n] + sum)        (out: [M][Nw])
//   kThinQkvRope   bias added, rounded to bf16, q and k heads rotated with the
//                  cos/sin table `rope` ([M][d/2] float2, scale applied), v
//                  copied, written in the [M][H][d] layouts of q, k, v
//   kThinSilu      out[m][j] = bf16(SiLU(bf16(gate)) bf16(up)) (out: [M][I];
//                  paired_I = I: gate rows [0, I), up rows [I, 2I) of W)
// The X tensor map's box is 64 x Mp, the W map's 64 x 128 (128-byte swizzle).
constexpr int kThinMaxRows = 256;
constexpr int kThinMaxSplits = 8;
enum ThinOp : int { kThinResidual = 0, kThinQkvRope = 1, kThinSilu = 2 };
struct ThinPlan {
    int tiles, k_steps, kps, splits, Mp, stages, wblocks;
    size_t region, smem;  // ring / staging bytes; dynamic shared memory of the launch
};
ThinPlan thin_plan(int M, int Nw, int K, int sms, int paired_I);
struct ThinParams {
    int M, Mp, Nw, K, k_steps, kps, splits, stages, paired_I, op, wblocks;
    size_t region;
    __nv_bfloat16* out;             // residual / silu output
    const __nv_bfloat16* bias;      // qkv: nullable [Nw]
    __nv_bfloat16 *q, *k, *v;       // qkv: [M][Hq][d], [M][Hkv][d], [M][Hkv][d]
    const float2* rope;             // qkv: [M][d / 2] (cos, sin)
    int Hq, Hkv, d;
    int32_t* status;
    unsigned long long watchdog_ns;
};
// Sets the kernel's shared-memory limit and measures, on the current device,
// how many clusters of each size fit at once (the plans use it).
cudaError_t thin_prepare();
cudaError_t launch_thin_gemm(const CUtensorMap& tm_x, const CUtensorMap& tm_w, const ThinParams& p,
                             size_t smem, cudaStream_t st);
// RMSNorm as launch_rmsnorm, and, when rp is set, the RoPE table of the next
// QKV projection: rope[r][k] = (cos, sin)(p * freq[k]) * scale for row r's
// virtual position p (the same fp64 angle and fp32 sin/cos as the rotation
// kernel).
cudaError_t launch_rmsnorm_rope(const __nv_bfloat16* x, const __nv_bfloat16* g, float eps,
                                __nv_bfloat16* y, int rows, int H, const RopeParams& rp, float2* rope,
                                cudaStream_t st);


// One-pass split-K decoding over the cache (decode_kernel.cu): for up to
// kDecodeRows query rows (new tokens x query heads of a KV head).
constexpr int kDecodeRows = 16;
constexpr int kDecodeMaxChunks = 64;
struct DecodeParams {
    const __nv_bfloat16* q;     // [U][n][Hq][D]
    __nv_bfloat16* out;         // [U][n][Hq][D]
    const __nv_bfloat16* cache_k;  // arena [S*L][Hkv][cap][D]
    const __nv_bfloat16* cache_v;
    const int32_t* frames;      // arena [S*L][Hkv]: rows before = frames * T + text
    const int32_t* text;
    float* part_o;              // [U][Hkv][nchunk][kDecodeRows][D]
    float* part_ml;             // [U][Hkv][nchunk][kDecodeRows][2]
    UnitRange units;
    int n, G, Hq, Hkv, T;
    long long cap;
    int ck, nchunk;             // keys per chunk (a multiple of 256), chunks
    float scale_log2;
    int32_t* status;
    unsigned long long watchdog_ns;
};
// tm_k / tm_v: the decode caches as 4-D maps [S*L][Hkv][cap][D] with boxes of
// 64 columns x 32 keys (kDecodeKeyBox), 128-byte swizzle
constexpr int kDecodeKeyBox = 32;
cudaError_t launch_decode(const CUtensorMap& tm_k, const CUtensorMap& tm_v, const DecodeParams& p, int D,
                          int U, cudaStream_t st);
cudaError_t decode_prepare();  // once, before the first launch_decode

// Recency-window state update (the baseline): the frame's tokens enter ring
// slots position mod B, overwriting the tokens that leave the window.
cudaError_t launch_recency(const RecencyParams& p, cudaStream_t st);

// Adds `n` to counter[unit_abs(u) * Hkv + h] for every unit u < U and head h.
cudaError_t launch_advance(int32_t* counter, UnitRange units, int U, int Hkv, int n,
                           cudaStream_t st);

// Shared-memory bytes the attention kernel needs for head dim D.
size_t attn_smem_bytes(int D);
// Largest pool (B + T) the select kernel keeps in shared memory, and the
// largest frame (T) it lists.
constexpr int kMaxPool = 24576;
constexpr int kMaxFrameTokens = 4096;
size_t select_smem_bytes(int P, int T);

// Every TMA descriptor of the library: a 4-D bf16 tensor map (dims and byte
// strides innermost first) with a (64, b1, b2, 1) box, 128-byte swizzle and
// zero fill out of bounds -- the layout the attention kernel's shared-memory
// descriptors assume.  False when the driver entry point is missing or the
// driver rejects the map.
bool encode_4d(CUtensorMap* m, const void* base, const cuuint64_t dims[4],
               const cuuint64_t strides_bytes[3], const cuuint32_t box[4]);
bool tma_encode_available();

cudaError_t attn_prepare(int D);
int device_sm_count();  // SMs of the current device (read by attn_prepare)
cudaError_t select_prepare();
cudaError_t launch_attn(int D, const CUtensorMap& tm_sk, const CUtensorMap& tm_sv,
                        const CUtensorMap& tm_fk, const CUtensorMap& tm_fv, const AttnParams& p,
                        int U, cudaStream_t st);
cudaError_t launch_select(const SelectParams& p, int U, cudaStream_t st);
cudaError_t launch_append(const AppendParams& p, cudaStream_t st);

// Debug builds: compares every byte of up to kMaxGuards 256-byte guard bands
// of the arena with the fill pattern kGuardFill; a mismatch records
// DEV_CANARY with the band's index.
constexpr int kMaxGuards = 24;
constexpr int kGuardBytes = 256;
constexpr unsigned char kGuardFill = 0xA5;
struct GuardList {
    unsigned long long off[kMaxGuards];
    int n;
};
cudaError_t launch_canary_check(const uint8_t* arena, const GuardList& g, int32_t* status, cudaStream_t st);

}  // namespace statekv
