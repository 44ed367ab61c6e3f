// The VLM's LLM prefill (App. A, Tab. "Model architecture parameters of pi series VLA models",
// Sec. 4.3): Gemma-shaped blocks over the prefix tokens, writing each layer's rotated keys and
// values straight into the action expert's KV store.
//
// The Q/K/V, output, gate/up and down projections are plain GEMMs with batch * prefix rows (816
// per request) on this file's tcgen05 GEMM (bf16 operands by bulk tensor copies, fp32
// accumulation in TMEM, see k_pf_gemm); the residual stream stays fp32 and the two residual
// projections accumulate into it in place. Attention (all heads stacked as query rows, since the
// single KV head is shared) runs on the expert's tcgen05 attention kernel with every key visible;
// for head dims or store strides that kernel does not take, it falls back to per-request GEMMs:
// the scores q K^T, a row softmax, V transposed, and the probabilities times V. This file's other
// kernels do the rest: RMSNorm to a bf16 operand, rotary coding of q and k from a table built
// once in double precision (with k and v scattered into the store), and GeGLU.

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <new>
#include <vector>

#include "jpi_prefill.h"
#include "../ptx.h"
#include "../attn_t5_kernel.cuh"

namespace {

thread_local char g_err[1024] = "";

jpi_status pfail(jpi_status s, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return s;
}

#define PF_CUDA(expr)                                                                              \
    do {                                                                                           \
        cudaError_t e_ = (expr);                                                                   \
        if (e_ != cudaSuccess)                                                                     \
            return pfail(JPI_ERR_CUDA, "%s failed: %s (%s:%d)", #expr, cudaGetErrorString(e_),     \
                         __FILE__, __LINE__);                                                      \
    } while (0)

#define PF_TRY(expr)                         \
    do {                                     \
        jpi_status s_ = (expr);              \
        if (s_ != JPI_OK) return s_;         \
    } while (0)

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) v += __shfl_xor_sync(0xffffffffu, v, s);
    return v;
}

__device__ __forceinline__ float gelu_tanh_f(float y) {
    // 0.5 y (1 + tanh(sqrt(2/pi) (y + 0.044715 y^3))), the tanh form of GELU.
    return 0.5f * y * (1.f + tanhf(0.7978845608028654f * (y + 0.044715f * y * y * y)));
}

__global__ void k_pf_cast(const float* __restrict__ src, __nv_bfloat16* __restrict__ dst, long long n) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x)
        dst[i] = __float2bfloat16_rn(src[i]);
}

// h = x (fp32 or bf16 embeddings) as the fp32 residual stream.
__global__ void k_pf_load_x(const void* __restrict__ x, int x_fp32, float* __restrict__ h, long long n) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x)
        h[i] = x_fp32 ? static_cast<const float*>(x)[i] : __bfloat162float(static_cast<const __nv_bfloat16*>(x)[i]);
}

// Row kernels of W floats (W a multiple of 4): one block of RB threads per row (grid-stride over
// rows), a row of up to RB x RB_CAP float4 held in registers with every load in flight, the sum
// of squares reduced over the block.
constexpr int RB = 128;
constexpr int RB_CAP = 8;   // 4096 floats per row
__device__ __forceinline__ float block_sum_rb(float v, float* red) {
    v = warp_sum(v);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    float t = 0.f;
#pragma unroll
    for (int i = 0; i < RB / 32; ++i) t += red[i];
    __syncthreads();   // red is reused by the next row
    return t;
}
// y[4 i .. 4 i + 3] of row r = v * rinv * (1 + w).
template <typename TO>
__device__ __forceinline__ void store_normed4(TO* y, const float* w, long long r, int W, int i, float4 v, float rinv) {
    const float4 g = reinterpret_cast<const float4*>(w)[i];
    const float a0 = v.x * rinv * (1.f + g.x), a1 = v.y * rinv * (1.f + g.y);
    const float a2 = v.z * rinv * (1.f + g.z), a3 = v.w * rinv * (1.f + g.w);
    if constexpr (sizeof(TO) == 2) {
        const __nv_bfloat162 lo = __floats2bfloat162_rn(a0, a1), hi = __floats2bfloat162_rn(a2, a3);
        uint2 u;
        u.x = *reinterpret_cast<const uint32_t*>(&lo);
        u.y = *reinterpret_cast<const uint32_t*>(&hi);
        *reinterpret_cast<uint2*>(y + r * W + 4 * i) = u;
    } else {
        *reinterpret_cast<float4*>(y + r * W + 4 * i) = make_float4(a0, a1, a2, a3);
    }
}
__device__ __forceinline__ float sq4(float4 v) {
    return (v.x * v.x + v.y * v.y) + (v.z * v.z + v.w * v.w);
}

// y = h / sqrt(mean(h^2) + eps) * (1 + w), row by row.
template <typename TO>
__global__ void __launch_bounds__(RB) k_pf_rmsnorm(const float* __restrict__ h, const float* __restrict__ w,
                                                   TO* __restrict__ y, long long rows, int W, float eps) {
    __shared__ float red[RB / 32];
    const int t = threadIdx.x, n4 = W >> 2;
    for (long long r = blockIdx.x; r < rows; r += gridDim.x) {
        const float4* hr = reinterpret_cast<const float4*>(h + r * W);
        if (n4 <= RB * RB_CAP) {
            float4 v[RB_CAP];
            float s = 0.f;
#pragma unroll
            for (int k = 0; k < RB_CAP; ++k) {
                const int i = t + RB * k;
                v[k] = i < n4 ? hr[i] : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int k = 0; k < RB_CAP; ++k) s += sq4(v[k]);
            const float rinv = 1.f / sqrtf(block_sum_rb(s, red) / (float)W + eps);
#pragma unroll
            for (int k = 0; k < RB_CAP; ++k) {
                const int i = t + RB * k;
                if (i < n4) store_normed4(y, w, r, W, i, v[k], rinv);
            }
        } else {
            float s = 0.f;
            for (int i = t; i < n4; i += RB) s += sq4(hr[i]);
            const float rinv = 1.f / sqrtf(block_sum_rb(s, red) / (float)W + eps);
            for (int i = t; i < n4; i += RB) store_normed4(y, w, r, W, i, hr[i], rinv);
        }
    }
}

// From the projections qkv [B P][(H + 2) D] (fp32): rotated queries q [B P][H][D] (bf16), and the
// rotated keys and the values of request b, row p into kd / vd + b stride + p D (bf16). One block
// per token row (grid-stride), its threads over the (section, rotary pair) slots of the row;
// rope[p][j] = (cos, sin) of p base^(-2j/D).
__global__ void k_pf_rope_scatter(const float* __restrict__ qkv, const float2* __restrict__ rope,
                                  __nv_bfloat16* __restrict__ q, __nv_bfloat16* __restrict__ kd,
                                  __nv_bfloat16* __restrict__ vd, long long stride, int B, int P, int H,
                                  int D) {
    const int half = D / 2, secs = H + 2, slots = secs * half;
    constexpr int RS_BATCH = 8;   // slots of a thread whose loads are in flight together
    for (long long r = blockIdx.x; r < (long long)B * P; r += gridDim.x) {   // r = b P + p
        const int p = (int)(r % P), b = (int)(r / P);
        const float* row = qkv + r * (long long)secs * D;
        for (int t0 = threadIdx.x; t0 < slots; t0 += RS_BATCH * blockDim.x) {
            float x1[RS_BATCH], x2[RS_BATCH];
            float2 cs[RS_BATCH];
#pragma unroll
            for (int u = 0; u < RS_BATCH; ++u) {
                const int t = t0 + u * blockDim.x;
                x1[u] = x2[u] = 0.f;
                cs[u] = make_float2(1.f, 0.f);
                if (t < slots) {
                    const int s = t / half, j = t - s * half;
                    const float* src = row + s * D;
                    x1[u] = src[j];
                    x2[u] = src[j + half];
                    if (s <= H) cs[u] = rope[(size_t)p * half + j];
                }
            }
#pragma unroll
            for (int u = 0; u < RS_BATCH; ++u) {
                const int t = t0 + u * blockDim.x;
                if (t >= slots) break;
                const int s = t / half, j = t - s * half;
                float y1 = x1[u], y2 = x2[u];
                if (s <= H) {
                    y1 = x1[u] * cs[u].x - x2[u] * cs[u].y;
                    y2 = x2[u] * cs[u].x + x1[u] * cs[u].y;
                }
                __nv_bfloat16* dst;
                if (s < H) dst = q + (r * H + s) * (long long)D;
                else dst = (s == H ? kd : vd) + b * stride + (long long)p * D;
                dst[j] = __float2bfloat16_rn(y1);
                dst[j + half] = __float2bfloat16_rn(y2);
            }
        }
    }
}

// probs[r][0 .. n) = softmax(s[r][0 .. n)) as bf16 (rows of stride ld); one warp per row. Rows of
// up to SM_CAP values per lane are read once into registers (all loads in flight together);
// longer rows take three strided passes.
constexpr int SM_CAP = 32;   // 1024 keys
__global__ void __launch_bounds__(256) k_pf_softmax(const float* __restrict__ s, __nv_bfloat16* __restrict__ p,
                                                    long long rows, int n, int ld) {
    const int lane = threadIdx.x & 31;
    const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
    for (long long r = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < rows; r += nwarps) {
        const float* sr = s + r * ld;
        __nv_bfloat16* pr = p + r * ld;
        if (n <= 32 * SM_CAP) {
            float v[SM_CAP];
            float mx = -INFINITY;
#pragma unroll
            for (int k = 0; k < SM_CAP; ++k) {
                const int j = lane + 32 * k;
                v[k] = j < n ? sr[j] : -INFINITY;
            }
#pragma unroll
            for (int k = 0; k < SM_CAP; ++k) mx = fmaxf(mx, v[k]);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
            float den = 0.f;
#pragma unroll
            for (int k = 0; k < SM_CAP; ++k) {
                v[k] = lane + 32 * k < n ? expf(v[k] - mx) : 0.f;
                den += v[k];
            }
            const float inv = 1.f / warp_sum(den);
#pragma unroll
            for (int k = 0; k < SM_CAP; ++k) {
                const int j = lane + 32 * k;
                if (j < n) pr[j] = __float2bfloat16_rn(v[k] * inv);
            }
        } else {
            float mx = -INFINITY;
            for (int j = lane; j < n; j += 32) mx = fmaxf(mx, sr[j]);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
            float den = 0.f;
            for (int j = lane; j < n; j += 32) den += expf(sr[j] - mx);
            const float inv = 1.f / warp_sum(den);
            for (int j = lane; j < n; j += 32) pr[j] = __float2bfloat16_rn(expf(sr[j] - mx) * inv);
        }
    }
}

// After a product split over K ranges: h += (part_0 + part_1 + ...) in range order (parts [rows][W]
// fp32, `pstride` elements apart), then, when w is set, the next RMSNorm y = h / sqrt(mean(h^2) +
// eps) * (1 + w) as k_pf_rmsnorm computes it.
template <typename TO>
__global__ void __launch_bounds__(RB) k_pf_residual_norm(float* __restrict__ h, const float* __restrict__ parts,
                                                         int nparts, long long pstride, const float* __restrict__ w,
                                                         TO* __restrict__ y, long long rows, int W, float eps) {
    __shared__ float red[RB / 32];
    const int t = threadIdx.x, n4 = W >> 2;
    for (long long r = blockIdx.x; r < rows; r += gridDim.x) {
        float4* hr = reinterpret_cast<float4*>(h + r * W);
        // h + (part_0 + part_1 + ...) for float4 i.
        auto update = [&](int i) {
            float4 d = reinterpret_cast<const float4*>(parts + r * W)[i];
            for (int q = 1; q < nparts; ++q) {
                const float4 e = reinterpret_cast<const float4*>(parts + (size_t)q * pstride + r * W)[i];
                d = make_float4(d.x + e.x, d.y + e.y, d.z + e.z, d.w + e.w);
            }
            const float4 o = hr[i];
            const float4 v = make_float4(o.x + d.x, o.y + d.y, o.z + d.z, o.w + d.w);
            hr[i] = v;
            return v;
        };
        if (n4 <= RB * RB_CAP) {
            // Passes over the row held in registers: part 0, each further part, then h.
            float4 v[RB_CAP];
            const float4* p0 = reinterpret_cast<const float4*>(parts + r * W);
#pragma unroll
            for (int k = 0; k < RB_CAP; ++k) {
                const int i = t + RB * k;
                v[k] = i < n4 ? p0[i] : make_float4(0.f, 0.f, 0.f, 0.f);
            }
            for (int q = 1; q < nparts; ++q) {
                const float4* pq = reinterpret_cast<const float4*>(parts + (size_t)q * pstride + r * W);
#pragma unroll
                for (int k = 0; k < RB_CAP; ++k) {
                    const int i = t + RB * k;
                    if (i < n4) {
                        const float4 e = pq[i];
                        v[k] = make_float4(v[k].x + e.x, v[k].y + e.y, v[k].z + e.z, v[k].w + e.w);
                    }
                }
            }
            // The residual row: every load before the stores that update it.
            float4 o[RB_CAP];
#pragma unroll
            for (int k = 0; k < RB_CAP; ++k) {
                const int i = t + RB * k;
                o[k] = i < n4 ? hr[i] : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int k = 0; k < RB_CAP; ++k) {
                const int i = t + RB * k;
                if (i < n4) {
                    v[k] = make_float4(o[k].x + v[k].x, o[k].y + v[k].y, o[k].z + v[k].z, o[k].w + v[k].w);
                    hr[i] = v[k];
                }
            }
            if (!w) continue;
            float s = 0.f;
#pragma unroll
            for (int k = 0; k < RB_CAP; ++k) s += sq4(v[k]);
            const float rinv = 1.f / sqrtf(block_sum_rb(s, red) / (float)W + eps);
#pragma unroll
            for (int k = 0; k < RB_CAP; ++k) {
                const int i = t + RB * k;
                if (i < n4) store_normed4(y, w, r, W, i, v[k], rinv);
            }
        } else {
            float s = 0.f;
            for (int i = t; i < n4; i += RB) s += sq4(update(i));
            if (!w) continue;
            const float rinv = 1.f / sqrtf(block_sum_rb(s, red) / (float)W + eps);
            for (int i = t; i < n4; i += RB) store_normed4(y, w, r, W, i, hr[i], rinv);
        }
    }
}

// Gate (off = 0) or up (off = 128) rows [F][W] fp32 -> bf16 rows of the packed gate/up matrix,
// where 256-row tile t holds gate rows 128 t..128 t + 127, then the up rows of the same features.
__global__ void k_pf_cast_gu(const float* __restrict__ src, __nv_bfloat16* __restrict__ dst, int F, int W, int off) {
    const long long n = (long long)F * W;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
        const int f = (int)(i / W), c = (int)(i - (long long)f * W);
        const long long row = (long long)(f >> 7) * 256 + off + (f & 127);
        dst[row * W + c] = __float2bfloat16_rn(src[i]);
    }
}

int grid_for(long long threads, int block = 256, int cap = 16384) {
    long long g = (threads + block - 1) / block;
    if (g < 1) g = 1;
    if (g > cap) g = cap;
    return (int)g;
}

struct LayerW {
    __nv_bfloat16 *wqkv = nullptr, *wo = nullptr, *wgu = nullptr, *wd = nullptr;
    float *attn_norm = nullptr, *mlp_norm = nullptr;
};

// ---------------------------------------------------------------------------------------------
// The products: Y[m][n] = alpha sum_k X[m][k] W[n][k] (+ Y[m][n]), X [M][K] and W [N][K] row-major
// bf16, Y fp32 or bf16, fp32 accumulation. One output tile = 128 rows of X (the MMA's M) x 256
// rows of W (its N) over the whole K range, in TMEM as [X row = lane][W row = column]: each k-block
// brings 48 KB into the SM for 2 M multiply-adds (a 128 x 128 tile brings 32 KB for 1 M, and one
// SM takes in only about 85 GB/s from L2), and only the token dimension, 816 rows at Gemma-2B
// sizes, is padded. Persistent: one CTA per SM walks the tiles u = blockIdx.x, + gridDim.x, ...
// with the X tile fastest, so the CTAs that run together share one W tile through L2 and every W
// tile is read from HBM once (W is the large operand: 134 MB for gate/up, X 3.3 MB):
//   warp 0  one thread streams (X block, W block) pairs of 64 K-columns by bulk tensor copies
//           (128-byte swizzle; rows and columns past the tensors' extents arrive as zeros) into a
//           ring of PG_STAGES stages;
//   warp 1  one thread issues the tcgen05.mma chain (M = 128, N = 256, K = 16 each) into one of two
//           TMEM accumulators and releases each stage through tcgen05.commit;
//   warps 2-5  one TMEM lane (X row m) per thread: 16 columns (W rows n) at a time, scaled by
//           alpha, added to Y when accumulating, stored as 16 consecutive elements of row m, after
//           which the accumulator goes back to the MMA thread.
// Every wait is bounded; a timeout records a device error in the handle's word and the CTA returns.

constexpr int PG_TM = 128;                                      // X rows per tile (MMA M)
constexpr int PG_TN = 256;                                      // W rows per tile (MMA N)
constexpr int PG_KBLK = 64;
constexpr int PG_STAGES = 4;
constexpr int PG_XBYTES = PG_TM * PG_KBLK * 2;                  // 16 KB
constexpr int PG_WBYTES = PG_TN * PG_KBLK * 2;                  // 32 KB
constexpr int PG_STAGE_BYTES = PG_XBYTES + PG_WBYTES;
constexpr int PG_THREADS = 192;
constexpr uint64_t PG_WAIT_NS = 200ull * 1000 * 1000;
constexpr size_t PG_SMEM = 1024 + (size_t)PG_STAGES * PG_STAGE_BYTES + 128;

enum PfDeviceError { PF_DEV_OK = 0, PF_DEV_TIMEOUT_LOAD = 1, PF_DEV_TIMEOUT_MMA = 2 };

struct PfGemmArgs {
    int M, N, K;          // K: columns the maps cover (a multiple of 64 is not required)
    float alpha;
    int accumulate;       // Y += ... (fp32 Y only)
    int out_bf16;
    int vec;              // Y and ldy allow 16-byte stores of 16 consecutive elements
    void* Y;
    long long ldy;        // elements
    // K split: k-blocks in ksplit consecutive ranges; range s writes its partial products to
    // Y + s * ysplit (fp32, never accumulating), summed in range order by the consumer.
    int ksplit;
    long long ysplit;
    // GeGLU: W tile t holds gate rows 128 t.. then the up rows of the same features; Y is bf16
    // z [M][ldy] = gelu_tanh(alpha gate) * (alpha up) for the nz features.
    int geglu, nz;
    int* err;
};

__global__ void __launch_bounds__(PG_THREADS, 1) k_pf_gemm(const __grid_constant__ CUtensorMap wmap,
                                                         const __grid_constant__ CUtensorMap xmap,
                                                         const __grid_constant__ PfGemmArgs a) {
    namespace ptx = jpi::ptx;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (ptx::smem_u32(smem_raw) & 1023u)) & 1023u);
    uint8_t* stages = smem;                                  // [stage][X 16 KB | W 32 KB]
    uint64_t* full = (uint64_t*)(smem + (size_t)PG_STAGES * PG_STAGE_BYTES);
    uint64_t* empty = full + PG_STAGES;
    uint64_t* accf = empty + PG_STAGES;
    uint64_t* acce = accf + 2;
    uint32_t* tmem_slot = (uint32_t*)(acce + 2);
    int* flag = (int*)(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int nkb = (a.K + PG_KBLK - 1) / PG_KBLK;
    const int ntn = (a.N + PG_TN - 1) / PG_TN, ntm = (a.M + PG_TM - 1) / PG_TM;
    const int total = ntn * ntm * a.ksplit;
    const int u0 = blockIdx.x, du = gridDim.x;
    // Unit u: X tile fastest, then W tile, then K range; k-blocks [kb_lo, kb_hi) of the range.
    const int nkr = (nkb + a.ksplit - 1) / a.ksplit;
    auto unit = [&](int u, int& tm, int& tn, int& sk, int& kb_lo, int& kb_hi) {
        tm = u % ntm;
        tn = (u / ntm) % ntn;
        sk = u / (ntm * ntn);
        kb_lo = sk * nkr;
        kb_hi = min(nkb, kb_lo + nkr);
    };

    if (warp == 1) {
        ptx::tmem_alloc(tmem_slot, 2 * PG_TN);
        ptx::tmem_relinquish();
    }
    if (tid == 0) {
        for (int i = 0; i < 2 * PG_STAGES; ++i) ptx::mbar_init(&full[i], 1);
        ptx::mbar_init(&accf[0], 1);
        ptx::mbar_init(&accf[1], 1);
        ptx::mbar_init(&acce[0], 128);
        ptx::mbar_init(&acce[1], 128);
        ptx::fence_mbar_init();
        *flag = 0;
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            int it = 0, issued = 0;
            bool ok = true;
            for (int u = u0; u < total && ok; u += du) {
                int tm, tn, sk, kb_lo, kb_hi;
                unit(u, tm, tn, sk, kb_lo, kb_hi);
                for (int kb = kb_lo; kb < kb_hi; ++kb, ++it) {
                    const int s = it % PG_STAGES, n = it / PG_STAGES;
                    if (it >= PG_STAGES && !ptx::mbar_wait_bounded(&empty[s], (n - 1) & 1, PG_WAIT_NS)) {
                        *flag = PF_DEV_TIMEOUT_LOAD;
                        ok = false;
                        break;
                    }
                    uint8_t* st = stages + (size_t)s * PG_STAGE_BYTES;
                    ptx::mbar_expect_tx(&full[s], (uint32_t)PG_STAGE_BYTES);
                    ptx::tma_load_2d_plain(st, &xmap, &full[s], kb * PG_KBLK, tm * PG_TM);
                    ptx::tma_load_2d_plain(st + PG_XBYTES, &wmap, &full[s], kb * PG_KBLK, tn * PG_TN);
                    issued = it + 1;
                }
            }
            // Nothing may land in this CTA's shared memory after it exits: wait for the last copy
            // into every stage (complete already unless a wait above gave up).
            for (int i = issued - PG_STAGES < 0 ? 0 : issued - PG_STAGES; i < issued; ++i)
                if (!ptx::mbar_wait_bounded(&full[i % PG_STAGES], (i / PG_STAGES) & 1, PG_WAIT_NS))
                    *flag = PF_DEV_TIMEOUT_LOAD;
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t IDESC = ptx::idesc_bf16_f32(PG_TM, PG_TN);
            const uint32_t base = ptx::smem_u32(stages);
            bool good = true;
            int it = 0;
            for (int u = u0, j = 0; u < total; u += du, ++j) {
                const int buf = j & 1;
                if (j >= 2 && !ptx::mbar_wait_bounded(&acce[buf], ((j - 2) >> 1) & 1, PG_WAIT_NS)) good = false;
                ptx::tc_fence_after();
                const uint32_t acc = tmem + (uint32_t)(buf * PG_TN);
                int tm, tn, sk, kb_lo, kb_hi;
                unit(u, tm, tn, sk, kb_lo, kb_hi);
                for (int kb = kb_lo; kb < kb_hi; ++kb, ++it) {
                    const int s = it % PG_STAGES, n = it / PG_STAGES;
                    if (good && !ptx::mbar_wait_bounded(&full[s], n & 1, PG_WAIT_NS)) good = false;
                    ptx::tc_fence_after();
                    if (good) {
                        const uint32_t x = base + (uint32_t)(s * PG_STAGE_BYTES), w = x + PG_XBYTES;
#pragma unroll
                        for (int kk = 0; kk < PG_KBLK / 16; ++kk)
                            ptx::mma_bf16(acc, ptx::desc_sw128(x + kk * 32), ptx::desc_sw128(w + kk * 32), IDESC,
                                          (kb != kb_lo) || (kk != 0));
                    }
                    ptx::mma_commit(&empty[s]);
                }
                // Committed even after a timeout so that the epilogue wakes up.
                ptx::mma_commit(&accf[buf]);
            }
            if (!good) *flag = PF_DEV_TIMEOUT_MMA;
        }
    } else {
        const int row = (warp & 3) * 32 + lane;   // TMEM lane: X row of the tile
        const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
        for (int u = u0, j = 0; u < total; u += du, ++j) {
            const int buf = j & 1;
            int tm, tn, sk, kb_lo, kb_hi;
            unit(u, tm, tn, sk, kb_lo, kb_hi);
            const bool ok = ptx::mbar_wait_bounded(&accf[buf], (j >> 1) & 1, PG_WAIT_NS) && *flag == 0;
            ptx::tc_fence_after();
            const int m = tm * PG_TM + row;
            const bool live = ok && m < a.M;
            if (a.geglu) {
                // Gate columns c0.. and up columns 128 + c0.. of this tile: 16 features of z.
                for (int c0 = 0; c0 < PG_TN / 2; c0 += 16) {
                    uint32_t rg[16], ru[16];
                    ptx::tmem_ld_x16(lane_base + (uint32_t)(buf * PG_TN + c0), rg);
                    ptx::tmem_ld_x16(lane_base + (uint32_t)(buf * PG_TN + PG_TN / 2 + c0), ru);
                    ptx::tmem_ld_wait();
                    const int f0 = tn * (PG_TN / 2) + c0;
                    if (!live || f0 >= a.nz) continue;
                    float v[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i)
                        v[i] = gelu_tanh_f(a.alpha * __uint_as_float(rg[i])) * (a.alpha * __uint_as_float(ru[i]));
                    __nv_bfloat16* z = static_cast<__nv_bfloat16*>(a.Y) + (size_t)m * a.ldy + f0;
                    if (a.vec && f0 + 16 <= a.nz) {
                        uint32_t p[8];
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            __nv_bfloat162 t = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
                            p[i] = *reinterpret_cast<uint32_t*>(&t);
                        }
                        reinterpret_cast<uint4*>(z)[0] = make_uint4(p[0], p[1], p[2], p[3]);
                        reinterpret_cast<uint4*>(z)[1] = make_uint4(p[4], p[5], p[6], p[7]);
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i)
                            if (f0 + i < a.nz) z[i] = __float2bfloat16_rn(v[i]);
                    }
                }
                ptx::tc_fence_before();
                ptx::mbar_arrive(&acce[buf]);
                if (!ok && lane == 0) *flag = PF_DEV_TIMEOUT_MMA;
                continue;
            }
            // K range sk writes its own partial (never accumulating).
            void* Yu = a.ksplit > 1 ? (void*)(static_cast<float*>(a.Y) + (size_t)sk * a.ysplit) : a.Y;
            const bool accum = a.accumulate && a.ksplit == 1;
            for (int c0 = 0; c0 < PG_TN; c0 += 16) {
                uint32_t r[16];
                ptx::tmem_ld_x16(lane_base + (uint32_t)(buf * PG_TN + c0), r);
                ptx::tmem_ld_wait();
                const int n0 = tn * PG_TN + c0;
                if (!live || n0 >= a.N) continue;
                float v[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) v[i] = a.alpha * __uint_as_float(r[i]);
                const size_t o = (size_t)m * a.ldy + n0;
                if (a.vec && n0 + 16 <= a.N) {
                    if (a.out_bf16) {
                        uint4* y = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(Yu) + o);
                        uint32_t p[8];
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            __nv_bfloat162 t = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
                            p[i] = *reinterpret_cast<uint32_t*>(&t);
                        }
                        y[0] = make_uint4(p[0], p[1], p[2], p[3]);
                        y[1] = make_uint4(p[4], p[5], p[6], p[7]);
                    } else {
                        float4* y = reinterpret_cast<float4*>(static_cast<float*>(Yu) + o);
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            float4 t = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                            if (accum) {
                                const float4 old = y[q];
                                t.x += old.x;
                                t.y += old.y;
                                t.z += old.z;
                                t.w += old.w;
                            }
                            y[q] = t;
                        }
                    }
                } else {
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        if (n0 + i >= a.N) continue;
                        if (a.out_bf16) {
                            static_cast<__nv_bfloat16*>(Yu)[o + i] = __float2bfloat16_rn(v[i]);
                        } else {
                            float* y = static_cast<float*>(Yu) + o + i;
                            *y = accum ? *y + v[i] : v[i];
                        }
                    }
                }
            }
            ptx::tc_fence_before();
            ptx::mbar_arrive(&acce[buf]);
            if (!ok && lane == 0) *flag = PF_DEV_TIMEOUT_MMA;
        }
    }

    if (tid == 0 && *flag != 0) atomicCAS(a.err, 0, *flag);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc(tmem, 2 * PG_TN);
}

// vt[d][p] = v[p][d] for one request (p < P), so that P V runs as a product of K-major operands.
__global__ void k_pf_transpose(const __nv_bfloat16* __restrict__ v, __nv_bfloat16* __restrict__ vt, int P, int D,
                               int ldt) {
    __shared__ __nv_bfloat16 t[32][33];
    const int p0 = blockIdx.x * 32, d0 = blockIdx.y * 32;
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int p = p0 + i, d = d0 + threadIdx.x;
        if (p < P && d < D) t[i][threadIdx.x] = v[(size_t)p * D + d];
    }
    __syncthreads();
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int d = d0 + i, p = p0 + threadIdx.x;
        if (p < P && d < D) vt[(size_t)d * ldt + p] = t[threadIdx.x][i];
    }
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        cudaDriverEntryPointQueryResult q;
        void* p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (PFN_cuTensorMapEncodeTiled_v12000)p;
    }
    return fn;
}

}  // namespace

struct jpi_prefill_handle {
    jpi_prefill_config cfg;
    int L = 0, W = 0, H = 0, D = 0, F = 0, QKV = 0, Bm = 0, Pm = 0, Pp = 0;
    std::vector<void*> allocs;
    size_t bytes = 0;
    std::vector<LayerW> layers;
    float* final_norm = nullptr;
    float2* rope = nullptr;          // [Pm][D / 2]
    float* h = nullptr;              // [Bm Pm][W] residual stream
    __nv_bfloat16* xn = nullptr;     // [Bm Pm][W] GEMM operand: normed h
    float* qkv = nullptr;            // [Bm Pm][(H + 2) D]
    __nv_bfloat16* q = nullptr;      // [Bm Pm][H][D]
    __nv_bfloat16* o = nullptr;      // [Bm Pm][H D]
    __nv_bfloat16* z = nullptr;      // [Bm Pm][F] GeGLU output (the gate/up product's epilogue)
    float* part = nullptr;           // partial products of a K-split projection
    long long part_elems = 0;        // floats `part` holds
    int Fp = 0;                      // F rounded up to 128: gate/up tiles of 128 features
    float* sc = nullptr;             // [H Pm][Pp] scores of one request
    __nv_bfloat16* pr = nullptr;     // [H Pm][Pp] probabilities of one request
    __nv_bfloat16* vt = nullptr;     // [D][Pp] one request's values, transposed
    int* dev_err = nullptr;          // device error word of the GEMM's bounded waits
    int num_sms = 0;
};

namespace {

template <typename T>
jpi_status pf_alloc(jpi_prefill_handle* h, T** p, size_t count) {
    void* q = nullptr;
    const size_t bytes = count * sizeof(T);
    const cudaError_t e = cudaMalloc(&q, bytes ? bytes : 16);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return pfail(JPI_ERR_OOM, "cudaMalloc(%zu bytes) failed: %s", bytes, cudaGetErrorString(e));
    }
    h->allocs.push_back(q);
    h->bytes += bytes;
    *p = static_cast<T*>(q);
    return JPI_OK;
}

void release(jpi_prefill_handle* h) {
    for (void* p : h->allocs) cudaFree(p);
    h->allocs.clear();
}

// 2D bf16 tensor map over a row-major [rows][cols] matrix of leading dimension ld (elements),
// 128-byte swizzle, boxes of 64 columns x box_rows rows; reads past the extents return zeros.
jpi_status make_map(const void* base, long long rows, long long cols, long long ld, int box_rows, CUtensorMap* map) {
    auto enc = get_encode();
    if (!enc) return pfail(JPI_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable from the driver");
    if ((reinterpret_cast<uintptr_t>(base) & 15) || (ld * 2) % 16)
        return pfail(JPI_ERR_INVALID_ARG, "a GEMM operand is not 16-byte aligned (address or row stride)");
    const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    const cuuint32_t box[2] = {(cuuint32_t)PG_KBLK, (cuuint32_t)box_rows};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
                           estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return pfail(JPI_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
    return JPI_OK;
}

// Y [M][N] (leading dimension ldy; fp32, or bf16 when y_bf16) = alpha X [M][K] W[N][K]^T, plus Y
// when accumulating. X and W are bf16 with leading dimensions ldx and ldw. With ksplit > 1 the
// k-blocks are cut into ksplit ranges and range s writes fp32 Y + s * ysplit (not accumulating);
// with nz > 0, Y is the bf16 GeGLU output z [M][ldy] of nz features (gate/up tiles packed).
jpi_status row_gemm(jpi_prefill_handle* h, cudaStream_t st, const __nv_bfloat16* X, long long ldx,
                    const __nv_bfloat16* Wm, long long ldw, void* Y, bool y_bf16, long long ldy, int M, int N,
                    int K, float alpha, bool accumulate, int ksplit = 1, long long ysplit = 0, int nz = 0) {
    CUtensorMap wmap, xmap;
    PF_TRY(make_map(Wm, N, K, ldw, PG_TN, &wmap));
    PF_TRY(make_map(X, M, K, ldx, PG_TM, &xmap));
    PfGemmArgs a;
    a.M = M;
    a.N = N;
    a.K = K;
    a.alpha = alpha;
    a.accumulate = accumulate ? 1 : 0;
    a.out_bf16 = y_bf16 ? 1 : 0;
    a.Y = Y;
    a.ldy = ldy;
    a.vec = (reinterpret_cast<uintptr_t>(Y) % 16 == 0 && ldy % (y_bf16 ? 8 : 4) == 0) ? 1 : 0;
    a.ksplit = ksplit;
    a.ysplit = ysplit;
    a.geglu = nz > 0 ? 1 : 0;
    a.nz = nz;
    a.err = h->dev_err;
    const long long tiles = (long long)((N + PG_TN - 1) / PG_TN) * ((M + PG_TM - 1) / PG_TM) * ksplit;
    const int grid = (int)(tiles < h->num_sms ? tiles : h->num_sms);
    k_pf_gemm<<<grid, PG_THREADS, PG_SMEM, st>>>(wmap, xmap, a);
    PF_CUDA(cudaGetLastError());
    return JPI_OK;
}

// K ranges for a product with few output tiles (at small B x P the O and down projections have
// 56 tiles at Gemma-2B sizes): as many as keep one wave on the GPU, at most 4, each of at least
// 8 k-blocks, and only while the partials [M][N] fit.
int split_for(const jpi_prefill_handle* h, int M, int N, int K) {
    const long long tiles = (long long)((N + PG_TN - 1) / PG_TN) * ((M + PG_TM - 1) / PG_TM);
    const int nkb = (K + PG_KBLK - 1) / PG_KBLK;
    int s = 1;
    while (s < 4 && tiles * (s + 1) <= h->num_sms && nkb / (s + 1) >= 8 &&
           (long long)(s + 1) * M * N <= h->part_elems)
        ++s;
    return s;
}

// Attention of the requests of one layer on the tcgen05 attention kernel: the queries h->q
// [B P H][D] against this layer's keys and values kd / vd (request b at row b * kv_rows, P rows
// each), every key visible, into h->o. Used for head dims 128 and 256 when the request stride is
// a whole number of rows; the maps' row extents end at the last request's last key, so no copy
// reads past what the caller owns (the kernel masks the zero-filled rows past P).
template <int D>
jpi_status attention_t5(jpi_prefill_handle* h, cudaStream_t st, const __nv_bfloat16* kd, const __nv_bfloat16* vd,
                        int batch, int P, long long kv_rows) {
    CUtensorMap qmap, kmap, vmap;
    const long long nrows = (long long)P * h->H;
    const long long krows = (long long)(batch - 1) * kv_rows + P;
    PF_TRY(make_map(h->q, (long long)batch * nrows, D, D, jpi::T5_ROWS, &qmap));
    PF_TRY(make_map(kd, krows, D, D, jpi::T5_KEYS, &kmap));
    PF_TRY(make_map(vd, krows, D, D, jpi::T5_KEYS, &vmap));
    jpi::T5Args a;
    a.S = P;
    a.nctx = 0;
    a.H = h->H;
    a.P = 0;
    a.kv_rows = (int)kv_rows;
    a.maxB = batch;
    a.layer = 0;
    a.scale_log2 = 1.4426950408889634f / sqrtf((float)D);
    a.o = h->o;
    a.err = h->dev_err;
    const dim3 grid((unsigned)((nrows + jpi::T5_ROWS - 1) / jpi::T5_ROWS), (unsigned)batch);
    jpi::k_attn_t5<D><<<grid, jpi::T5_THREADS, 1024 + jpi::T5Smem<D>::TOTAL, st>>>(qmap, kmap, vmap, a);
    PF_CUDA(cudaGetLastError());
    return JPI_OK;
}

jpi_status check_config(const jpi_prefill_config* c) {
    if (c->n_layers < 1 || c->n_heads < 1 || c->max_batch < 1 || c->max_prefix < 1)
        return pfail(JPI_ERR_INVALID_ARG, "n_layers, n_heads, max_batch and max_prefix must be >= 1");
    if (c->width < 8 || c->width % 8 || c->mlp_dim < 8 || c->mlp_dim % 8)
        return pfail(JPI_ERR_UNSUPPORTED, "width and mlp_dim must be multiples of 8");
    if (c->head_dim < 8 || c->head_dim % 8 || c->head_dim > 512)
        return pfail(JPI_ERR_UNSUPPORTED, "head_dim must be a multiple of 8 and at most 512");
    if ((long long)c->max_batch * c->max_prefix > (1ll << 24) || c->max_prefix > 65536)
        return pfail(JPI_ERR_UNSUPPORTED, "max_batch * max_prefix or max_prefix too large");
    if (!(c->rms_eps >= 0.f) || !(c->rope_base >= 0.f))
        return pfail(JPI_ERR_INVALID_ARG, "rms_eps and rope_base must be >= 0");
    return JPI_OK;
}

// fp32 tensor (host or device) -> bf16 at dst.
jpi_status put_bf16(jpi_prefill_handle* h, bool dev, float* staging, __nv_bfloat16* dst, const float* src,
                    size_t n, const char* name, int layer) {
    if (!src) return pfail(JPI_ERR_INVALID_ARG, "weight %s of layer %d is NULL", name, layer);
    const float* s = src;
    if (!dev) {
        PF_CUDA(cudaMemcpy(staging, src, n * sizeof(float), cudaMemcpyHostToDevice));
        s = staging;
    }
    k_pf_cast<<<grid_for((long long)n), 256>>>(s, dst, (long long)n);
    PF_CUDA(cudaGetLastError());
    // The staging buffer is reused by the next tensor; finish this conversion first.
    PF_CUDA(cudaStreamSynchronize(nullptr));
    return JPI_OK;
}

// Gate (off 0) or up (off 128) rows [F][W] (host or device fp32) into the packed gate/up matrix.
jpi_status put_gu(jpi_prefill_handle* h, bool dev, float* staging, __nv_bfloat16* dst, const float* src, int off,
                  const char* name, int layer) {
    if (!src) return pfail(JPI_ERR_INVALID_ARG, "weight %s of layer %d is NULL", name, layer);
    const size_t n = (size_t)h->F * h->W;
    const float* s = src;
    if (!dev) {
        PF_CUDA(cudaMemcpy(staging, src, n * sizeof(float), cudaMemcpyHostToDevice));
        s = staging;
    }
    k_pf_cast_gu<<<grid_for((long long)n), 256>>>(s, dst, h->F, h->W, off);
    PF_CUDA(cudaGetLastError());
    PF_CUDA(cudaStreamSynchronize(nullptr));
    return JPI_OK;
}

jpi_status put_f32(jpi_prefill_handle* h, bool dev, float** dst, const float* src, size_t n, const char* name,
                   int layer) {
    if (!src) return pfail(JPI_ERR_INVALID_ARG, "weight %s of layer %d is NULL", name, layer);
    PF_TRY(pf_alloc(h, dst, n));
    PF_CUDA(cudaMemcpy(*dst, src, n * sizeof(float), dev ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice));
    return JPI_OK;
}

jpi_status setup(jpi_prefill_handle* h, const jpi_prefill_config* c, const jpi_prefill_weights* w) {
    h->cfg = *c;
    h->L = c->n_layers;
    h->W = c->width;
    h->H = c->n_heads;
    h->D = c->head_dim;
    h->F = c->mlp_dim;
    h->QKV = (h->H + 2) * h->D;
    h->Bm = c->max_batch;
    h->Pm = c->max_prefix;
    h->Pp = (h->Pm + 7) / 8 * 8;
    const size_t W = (size_t)h->W, D = (size_t)h->D, F = (size_t)h->F, HD = (size_t)h->H * D;
    const size_t Mm = (size_t)h->Bm * h->Pm;
    h->Fp = (h->F + 127) / 128 * 128;
    const size_t Fp = (size_t)h->Fp;
    const bool dev = w->on_device != 0;
    if (!w->attn_norm || !w->wq || !w->wk || !w->wv || !w->wo || !w->mlp_norm || !w->w_gate || !w->w_up ||
        !w->w_down || !w->final_norm)
        return pfail(JPI_ERR_INVALID_ARG, "a weight array is NULL");

    int device = 0;
    PF_CUDA(cudaGetDevice(&device));
    PF_CUDA(cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, device));
    PF_CUDA(cudaFuncSetAttribute(k_pf_gemm, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)PG_SMEM));
    PF_CUDA(cudaFuncSetAttribute(jpi::k_attn_t5<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 1024 + jpi::T5Smem<128>::TOTAL));
    PF_CUDA(cudaFuncSetAttribute(jpi::k_attn_t5<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 1024 + jpi::T5Smem<256>::TOTAL));
    PF_TRY(pf_alloc(h, &h->dev_err, 1));
    PF_CUDA(cudaMemset(h->dev_err, 0, sizeof(int)));
    float* staging = nullptr;
    if (!dev) PF_TRY(pf_alloc(h, &staging, F * W));
    h->layers.resize((size_t)h->L);
    for (int l = 0; l < h->L; ++l) {
        LayerW& lw = h->layers[(size_t)l];
        PF_TRY(pf_alloc(h, &lw.wqkv, (HD + 2 * D) * W));
        PF_TRY(put_bf16(h, dev, staging, lw.wqkv, w->wq[l], HD * W, "wq", l));
        PF_TRY(put_bf16(h, dev, staging, lw.wqkv + HD * W, w->wk[l], D * W, "wk", l));
        PF_TRY(put_bf16(h, dev, staging, lw.wqkv + (HD + D) * W, w->wv[l], D * W, "wv", l));
        PF_TRY(pf_alloc(h, &lw.wo, W * HD));
        PF_TRY(put_bf16(h, dev, staging, lw.wo, w->wo[l], W * HD, "wo", l));
        PF_TRY(pf_alloc(h, &lw.wgu, 2 * Fp * W));
        PF_CUDA(cudaMemset(lw.wgu, 0, 2 * Fp * W * sizeof(__nv_bfloat16)));   // rows of features past F
        PF_TRY(put_gu(h, dev, staging, lw.wgu, w->w_gate[l], 0, "w_gate", l));
        PF_TRY(put_gu(h, dev, staging, lw.wgu, w->w_up[l], 128, "w_up", l));
        PF_TRY(pf_alloc(h, &lw.wd, W * F));
        PF_TRY(put_bf16(h, dev, staging, lw.wd, w->w_down[l], W * F, "w_down", l));
        PF_TRY(put_f32(h, dev, &lw.attn_norm, w->attn_norm[l], W, "attn_norm", l));
        PF_TRY(put_f32(h, dev, &lw.mlp_norm, w->mlp_norm[l], W, "mlp_norm", l));
    }
    PF_TRY(put_f32(h, dev, &h->final_norm, w->final_norm, W, "final_norm", -1));

    // Rotary table, in double precision on the host: angle p base^(-2j/D) for p < Pm, j < D/2.
    std::vector<float2> tab((size_t)h->Pm * (D / 2));
    for (int p = 0; p < h->Pm; ++p)
        for (size_t j = 0; j < D / 2; ++j) {
            float2 cs = make_float2(1.f, 0.f);
            if (c->rope_base > 0.f) {
                const double ang = (double)p * std::pow((double)c->rope_base, -2.0 * (double)j / (double)D);
                cs = make_float2((float)std::cos(ang), (float)std::sin(ang));
            }
            tab[(size_t)p * (D / 2) + j] = cs;
        }
    PF_TRY(pf_alloc(h, &h->rope, tab.size()));
    PF_CUDA(cudaMemcpy(h->rope, tab.data(), tab.size() * sizeof(float2), cudaMemcpyHostToDevice));

    PF_TRY(pf_alloc(h, &h->h, Mm * W));
    PF_TRY(pf_alloc(h, &h->xn, Mm * W));
    PF_TRY(pf_alloc(h, &h->z, Mm * F));
    // Partials of K-split projections (N = W): a split needs at most num_sms / 2 output tiles,
    // so a part has at most that many 128-row tiles of rows, and there are at most 4 parts.
    {
        const long long ntn = (h->W + PG_TN - 1) / PG_TN;
        const long long rows2 = std::min<long long>((long long)Mm, (h->num_sms / 2 / ntn) * PG_TM);
        h->part_elems = 4 * rows2 * h->W;
        if (h->part_elems > 0) PF_TRY(pf_alloc(h, &h->part, (size_t)h->part_elems));
    }
    PF_TRY(pf_alloc(h, &h->qkv, Mm * (size_t)h->QKV));
    PF_TRY(pf_alloc(h, &h->q, Mm * HD));
    PF_TRY(pf_alloc(h, &h->o, Mm * HD));
    PF_TRY(pf_alloc(h, &h->sc, (size_t)h->H * h->Pm * h->Pp));
    PF_TRY(pf_alloc(h, &h->pr, (size_t)h->H * h->Pm * h->Pp));
    PF_TRY(pf_alloc(h, &h->vt, D * (size_t)h->Pp));
    return JPI_OK;
}

}  // namespace

extern "C" {

JPI_API const char* jpi_prefill_last_error(void) { return g_err; }

JPI_API jpi_status jpi_prefill_create(const jpi_prefill_config* cfg, const jpi_prefill_weights* w,
                                      jpi_prefill_handle** out) {
    g_err[0] = '\0';
    if (!out) return pfail(JPI_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    if (!cfg || !w) return pfail(JPI_ERR_INVALID_ARG, "config or weights is NULL");
    PF_TRY(check_config(cfg));
    jpi_prefill_handle* h = new (std::nothrow) jpi_prefill_handle();
    if (!h) return pfail(JPI_ERR_OOM, "host allocation failed");
    const jpi_status s = setup(h, cfg, w);
    if (s != JPI_OK) {
        cudaStreamSynchronize(nullptr);
        cudaGetLastError();
        release(h);
        delete h;
        return s;
    }
    *out = h;
    return JPI_OK;
}

JPI_API jpi_status jpi_prefill_destroy(jpi_prefill_handle* h) {
    g_err[0] = '\0';
    if (!h) return JPI_OK;
    release(h);
    delete h;
    return JPI_OK;
}

JPI_API jpi_status jpi_prefill_run(jpi_prefill_handle* h, const void* x, int x_is_fp32, int batch, int prefix_len,
                                   void* const* k_layers, void* const* v_layers, long long request_stride,
                                   float* out_final, void* stream) {
    g_err[0] = '\0';
    if (!h) return pfail(JPI_ERR_INVALID_ARG, "handle is NULL");
    if (!x || !k_layers || !v_layers) return pfail(JPI_ERR_INVALID_ARG, "NULL input or KV destination array");
    if (batch < 1 || prefix_len < 1) return pfail(JPI_ERR_INVALID_ARG, "batch and prefix_len must be >= 1");
    if (batch > h->Bm || prefix_len > h->Pm)
        return pfail(JPI_ERR_SHAPE, "batch %d / prefix_len %d exceed the maxima %d / %d", batch, prefix_len, h->Bm,
                     h->Pm);
    if (request_stride < (long long)prefix_len * h->D || request_stride % 8)
        return pfail(JPI_ERR_INVALID_ARG, "request_stride must be >= prefix_len * head_dim and a multiple of 8");
    for (int l = 0; l < h->L; ++l)
        if (!k_layers[l] || !v_layers[l]) return pfail(JPI_ERR_INVALID_ARG, "KV destination of layer %d is NULL", l);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int W = h->W, D = h->D, H = h->H, F = h->F, P = prefix_len, Pp = (P + 7) / 8 * 8;
    const long long M = (long long)batch * P;
    const float eps = h->cfg.rms_eps, scale = 1.f / sqrtf((float)D);

    k_pf_load_x<<<grid_for(M * W), 256, 0, st>>>(x, x_is_fp32, h->h, M * W);
    PF_CUDA(cudaGetLastError());
    // After a K-split down projection, the step that adds its partials to h also writes the next
    // layer's attention norm into xn.
    bool xn_ready = false;
    const long long pstride = M * W;   // elements between the parts of a split product
    for (int l = 0; l < h->L; ++l) {
        const LayerW& lw = h->layers[(size_t)l];
        __nv_bfloat16* kd = static_cast<__nv_bfloat16*>(k_layers[l]);
        __nv_bfloat16* vd = static_cast<__nv_bfloat16*>(v_layers[l]);
        // Attention sublayer.
        if (!xn_ready) {
            k_pf_rmsnorm<__nv_bfloat16><<<grid_for(M, 1, 16384), RB, 0, st>>>(h->h, lw.attn_norm, h->xn, M, W, eps);
            PF_CUDA(cudaGetLastError());
        }
        PF_TRY(row_gemm(h, st, h->xn, W, lw.wqkv, W, h->qkv, false, h->QKV, (int)M, h->QKV, W, 1.f, false));
        k_pf_rope_scatter<<<grid_for(M, 1, 16384), 256, 0, st>>>(h->qkv, h->rope, h->q, kd, vd,
                                                                             request_stride, batch, P, H, D);
        PF_CUDA(cudaGetLastError());
        // Attention: on the tcgen05 attention kernel (scores and probabilities never leave the
        // SM), else per request through the GEMM: scores, softmax, V^T, probabilities times V.
        const bool t5 = (D == 128 || D == 256) && request_stride % D == 0 && request_stride / D <= INT32_MAX;
        if (t5) {
            PF_TRY(D == 256 ? attention_t5<256>(h, st, kd, vd, batch, P, request_stride / D)
                            : attention_t5<128>(h, st, kd, vd, batch, P, request_stride / D));
        }
        for (int b = 0; b < batch && !t5; ++b) {
            const __nv_bfloat16* qb = h->q + (size_t)b * P * H * D;     // [(P H)][D]
            const __nv_bfloat16* kb = kd + (size_t)b * request_stride;  // [P][D]
            const __nv_bfloat16* vb = vd + (size_t)b * request_stride;  // [P][D]
            __nv_bfloat16* ob = h->o + (size_t)b * P * H * D;           // [(P H)][D] = [P][H D]
            PF_TRY(row_gemm(h, st, qb, D, kb, D, h->sc, false, Pp, P * H, P, D, scale, false));
            k_pf_softmax<<<grid_for((long long)P * H * 32), 256, 0, st>>>(h->sc, h->pr, (long long)P * H, P, Pp);
            PF_CUDA(cudaGetLastError());
            k_pf_transpose<<<dim3((P + 31) / 32, (D + 31) / 32), dim3(32, 8), 0, st>>>(vb, h->vt, P, D, Pp);
            PF_CUDA(cudaGetLastError());
            PF_TRY(row_gemm(h, st, h->pr, Pp, h->vt, Pp, ob, true, D, P * H, D, P, 1.f, false));
        }
        // Output projection into the residual stream, then the MLP norm: split over K when the
        // product has too few tiles to fill the GPU (partials added in order with the norm).
        const int so = split_for(h, (int)M, W, H * D);
        if (so > 1) {
            PF_TRY(row_gemm(h, st, h->o, H * D, lw.wo, H * D, h->part, false, W, (int)M, W, H * D, 1.f, false, so,
                            pstride));
            k_pf_residual_norm<__nv_bfloat16><<<grid_for(M, 1, 16384), RB, 0, st>>>(h->h, h->part, so, pstride,
                                                                                  lw.mlp_norm, h->xn, M, W, eps);
        } else {
            PF_TRY(row_gemm(h, st, h->o, H * D, lw.wo, H * D, h->h, false, W, (int)M, W, H * D, 1.f, true));
            k_pf_rmsnorm<__nv_bfloat16><<<grid_for(M, 1, 16384), RB, 0, st>>>(h->h, lw.mlp_norm, h->xn, M, W, eps);
        }
        PF_CUDA(cudaGetLastError());
        // MLP sublayer: gate/up with GeGLU in its epilogue (z bf16), then down into the residual.
        PF_TRY(row_gemm(h, st, h->xn, W, lw.wgu, W, h->z, true, F, (int)M, 2 * h->Fp, W, 1.f, false, 1, 0, F));
        const int sd = split_for(h, (int)M, W, F);
        if (sd > 1) {
            PF_TRY(row_gemm(h, st, h->z, F, lw.wd, F, h->part, false, W, (int)M, W, F, 1.f, false, sd, pstride));
            if (l + 1 < h->L) {
                k_pf_residual_norm<__nv_bfloat16><<<grid_for(M, 1, 16384), RB, 0, st>>>(
                    h->h, h->part, sd, pstride, h->layers[(size_t)l + 1].attn_norm, h->xn, M, W, eps);
                xn_ready = true;
            } else if (out_final) {
                k_pf_residual_norm<float><<<grid_for(M, 1, 16384), RB, 0, st>>>(h->h, h->part, sd, pstride,
                                                                            h->final_norm, out_final, M, W, eps);
            } else {
                k_pf_residual_norm<float><<<grid_for(M, 1, 16384), RB, 0, st>>>(h->h, h->part, sd, pstride, nullptr,
                                                                            nullptr, M, W, eps);
            }
        } else {
            PF_TRY(row_gemm(h, st, h->z, F, lw.wd, F, h->h, false, W, (int)M, W, F, 1.f, true));
            xn_ready = false;
            if (l + 1 == h->L && out_final)
                k_pf_rmsnorm<float><<<grid_for(M, 1, 16384), RB, 0, st>>>(h->h, h->final_norm, out_final, M, W, eps);
        }
        PF_CUDA(cudaGetLastError());
    }
    return JPI_OK;
}

JPI_API jpi_status jpi_prefill_device_status(jpi_prefill_handle* h) {
    g_err[0] = '\0';
    if (!h) return pfail(JPI_ERR_INVALID_ARG, "handle is NULL");
    PF_CUDA(cudaDeviceSynchronize());
    int err = 0;
    PF_CUDA(cudaMemcpy(&err, h->dev_err, sizeof(int), cudaMemcpyDeviceToHost));
    if (err != PF_DEV_OK) {
        PF_CUDA(cudaMemset(h->dev_err, 0, sizeof(int)));
        return pfail(JPI_ERR_DEVICE_TIMEOUT, "device-side error code %d (a bounded wait in a product gave up)", err);
    }
    return JPI_OK;
}

JPI_API jpi_status jpi_prefill_memory_usage(const jpi_prefill_handle* h, long long* bytes) {
    g_err[0] = '\0';
    if (!h || !bytes) return pfail(JPI_ERR_INVALID_ARG, "handle or bytes is NULL");
    *bytes = (long long)h->bytes;
    return JPI_OK;
}

}  // extern "C"
