// The future correction module and its Q-Former state compressor on the GPU (Sec. 4.1, App. B
// and its figure, Eq. 2, App. C Alg. 1).
//
// Every token count here is small (T' = 4 compressed tokens, at most 64 committed actions per
// request), so apart from the compressor's pass over the VLM tokens the module is a chain of
// matrix-vector products that stream its ~44M weights once per call: at batch 1 that is HBM
// work (88 MB in bf16), not a dense contraction, and it runs on CUDA cores with every weight
// row read once by one warp (16-byte loads) and the few activation rows served from L1.
//
// The compressor's cross-attention is reassociated. Its queries come from the learned query
// tokens through the query self-attention alone, so they are fixed by the weights; with
// q_hi the scaled query of head h, item i, and W_k,h / W_v,h the head's rows of the key and
// value projections:
//   score_hij = q_hi . (W_k,h v_j + b_k,h) = (W_k,h^T q_hi) . v_j + const_hi,
//   out_hi    = sum_j p_hij (W_v,h v_j + b_v,h) = W_v,h (sum_j p_hij v_j) + b_v,h   (sum_j p = 1).
// The key bias only shifts every score of a query alike, which softmax cancels. So create time
// computes a_hi = W_k,h^T q_hi once ([H T'][d_vlm]); a call scores the raw VLM tokens against
// them, takes the softmax-weighted sum of the raw tokens, and applies W_v,h to that sum: about
// 2 H T' T d_vlm * 2 FLOPs per request instead of the 4 T d_vlm d of projecting every token.

#include "jpi_internal.h"
#include "ptx.h"

#include <map>
#include <tuple>
#include "jpi_corr.h"

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <new>
#include <utility>

namespace {

constexpr int CORR_MAX_M = 64;          // n_heads * n_items: rows of the reassociated queries
constexpr int LIN_ROWS = 8;             // activation rows one warp carries per weight-row pass

jpi_status cfail(jpi_status s, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    jpi::set_error("%s", buf);
    return s;
}

__device__ __forceinline__ float gelu_tanh_f(float y) {
    // 0.5 y (1 + tanh(sqrt(2/pi) (y + 0.044715 y^3))), the tanh form of GELU.
    return 0.5f * y * (1.f + tanhf(0.7978845608028654f * (y + 0.044715f * y * y * y)));
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) v += __shfl_xor_sync(0xffffffffu, v, s);
    return v;
}

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }

__device__ __forceinline__ float4 load4(const float* p) { return __ldg(reinterpret_cast<const float4*>(p)); }
__device__ __forceinline__ float4 load4(const __nv_bfloat16* p) {
    const uint2 u = __ldg(reinterpret_cast<const uint2*>(p));
    const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
    const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
    return make_float4(a.x, a.y, b.x, b.y);
}
__device__ __forceinline__ float load1(const float* p) { return __ldg(p); }
__device__ __forceinline__ float load1(const __nv_bfloat16* p) { return __bfloat162float(p[0]); }

// y[r][o] = act(sum_i x(r, o)[i] w[o][i] + bias[o]) + res[r][o] for r < rows, o < out.
// x(r, o) is row r of x (stride ldx), or in head-select mode row
// ((r / hs_items) * hs_heads + o / hs_dh) * hs_items + r % hs_items: the reassociated
// cross-attention keeps one weighted token sum per (request, head, item).
// One warp per output feature at a time; LIN_ROWS rows per pass over the weight row. y must not
// overlap x; it may be res (each element is read and written by the same lane).
struct LinArgs {
    const float* x;
    int ldx;
    const void* w;
    const float* bias;
    const float* res;
    int ldr;
    float* y;
    int ldy;
    int rows, in, out, gelu;
    int hs_items, hs_heads, hs_dh;   // head-select mode when hs_items > 0
};

template <typename TW, bool VEC>
__global__ void __launch_bounds__(256) k_corr_linear(const LinArgs a) {
    // Launched with programmatic dependent launch: wait for the previous kernel's results, then
    // let the next kernel's CTAs be scheduled (they wait in turn).
    jpi::ptx::grid_dep_wait();
    jpi::ptx::grid_dep_launch();
    const int lane = threadIdx.x & 31;
    const int nwarps = (gridDim.x * blockDim.x) >> 5;
    const TW* W = static_cast<const TW*>(a.w);
    for (int o = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5); o < a.out; o += nwarps) {
        const TW* wr = W + (size_t)o * a.in;
        const float bo = a.bias ? a.bias[o] : 0.f;
        for (int r0 = 0; r0 < a.rows; r0 += LIN_ROWS) {
            const float* xr[LIN_ROWS];
#pragma unroll
            for (int k = 0; k < LIN_ROWS; ++k) {
                const int r = r0 + k < a.rows ? r0 + k : a.rows - 1;   // clamped; result unused
                long long row = r;
                if (a.hs_items > 0)
                    row = ((long long)(r / a.hs_items) * a.hs_heads + o / a.hs_dh) * a.hs_items + r % a.hs_items;
                xr[k] = a.x + row * a.ldx;
            }
            float acc[LIN_ROWS];
#pragma unroll
            for (int k = 0; k < LIN_ROWS; ++k) acc[k] = 0.f;
            if (VEC) {
                // Unrolled so that several 4-wide weight loads of the row are in flight at once.
#pragma unroll 4
                for (int i = lane * 4; i < a.in; i += 128) {
                    const float4 w4 = load4(wr + i);
#pragma unroll
                    for (int k = 0; k < LIN_ROWS; ++k) {
                        const float4 x4 = *reinterpret_cast<const float4*>(xr[k] + i);
                        acc[k] = fmaf(w4.x, x4.x, fmaf(w4.y, x4.y, fmaf(w4.z, x4.z, fmaf(w4.w, x4.w, acc[k]))));
                    }
                }
            } else {
                for (int i = lane; i < a.in; i += 32) {
                    const float w1 = load1(wr + i);
#pragma unroll
                    for (int k = 0; k < LIN_ROWS; ++k) acc[k] = fmaf(w1, xr[k][i], acc[k]);
                }
            }
            float mine = 0.f;   // lane k keeps row r0 + k
#pragma unroll
            for (int k = 0; k < LIN_ROWS; ++k) {
                const float v = warp_sum(acc[k]);
                if (lane == k) mine = v;
            }
            const int r = r0 + lane;
            if (lane < LIN_ROWS && r < a.rows) {
                float v = mine + bo;
                if (a.gelu) v = gelu_tanh_f(v);
                if (a.res) v += a.res[(size_t)r * a.ldr + o];
                a.y[(size_t)r * a.ldy + o] = v;
            }
        }
    }
}

// The same product for bf16 weights with 16-byte aligned rows and 16-byte aligned activation rows
// (in a multiple of 8 KS, ldx of 4): a lane streams 16-byte weight chunks, LIN_CH of them in
// flight, and the KS consecutive warps of a block share an output feature, each over in / KS
// inputs, their sums added in warp order through shared memory (deterministic). Blocks of
// 8 / KS output features walk the outputs grid-stride.
constexpr int LIN_CH = 8;
template <int KS>
__global__ void __launch_bounds__(256) k_corr_linear16(const LinArgs a) {
    // Launched with programmatic dependent launch: wait for the previous kernel's results, then
    // let the next kernel's CTAs be scheduled (they wait in turn).
    jpi::ptx::grid_dep_wait();
    jpi::ptx::grid_dep_launch();
    __shared__ float part[8][LIN_ROWS];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int slice = warp % KS, og = warp / KS;
    constexpr int OPB = 8 / KS;
    const int kper = a.in / KS, k0 = slice * kper;
    const __nv_bfloat16* W = static_cast<const __nv_bfloat16*>(a.w);
    const int ngroups = (a.out + OPB - 1) / OPB;
    for (int gi = blockIdx.x; gi < ngroups; gi += gridDim.x) {
        const int o = gi * OPB + og;
        const bool live = o < a.out;
        const int oc = live ? o : a.out - 1;   // clamped; result unused
        const __nv_bfloat16* wr = W + (size_t)oc * a.in + k0;
        const float bo = (a.bias && live) ? a.bias[oc] : 0.f;
        for (int r0 = 0; r0 < a.rows; r0 += LIN_ROWS) {
            const float* xr[LIN_ROWS];
#pragma unroll
            for (int k = 0; k < LIN_ROWS; ++k) {
                const int r = r0 + k < a.rows ? r0 + k : a.rows - 1;   // clamped; result unused
                long long row = r;
                if (a.hs_items > 0)
                    row = ((long long)(r / a.hs_items) * a.hs_heads + oc / a.hs_dh) * a.hs_items + r % a.hs_items;
                xr[k] = a.x + row * a.ldx + k0;
            }
            float acc[LIN_ROWS];
#pragma unroll
            for (int k = 0; k < LIN_ROWS; ++k) acc[k] = 0.f;
            for (int base = 0; base < kper; base += 256 * LIN_CH) {
                uint4 wv[LIN_CH];
#pragma unroll
                for (int j = 0; j < LIN_CH; ++j) {
                    const int i = base + 256 * j + 8 * lane;
                    wv[j] = i < kper ? __ldg(reinterpret_cast<const uint4*>(wr + i)) : make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
                for (int j = 0; j < LIN_CH; ++j) {
                    const int i = base + 256 * j + 8 * lane;
                    if (i < kper) {
                        const uint32_t u[4] = {wv[j].x, wv[j].y, wv[j].z, wv[j].w};
                        float w[8];
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u[q]));
                            w[2 * q] = f.x;
                            w[2 * q + 1] = f.y;
                        }
#pragma unroll
                        for (int k = 0; k < LIN_ROWS; ++k) {
                            const float4 x0 = *reinterpret_cast<const float4*>(xr[k] + i);
                            const float4 x1 = *reinterpret_cast<const float4*>(xr[k] + i + 4);
                            float t = acc[k];
                            t = fmaf(w[0], x0.x, t);
                            t = fmaf(w[1], x0.y, t);
                            t = fmaf(w[2], x0.z, t);
                            t = fmaf(w[3], x0.w, t);
                            t = fmaf(w[4], x1.x, t);
                            t = fmaf(w[5], x1.y, t);
                            t = fmaf(w[6], x1.z, t);
                            t = fmaf(w[7], x1.w, t);
                            acc[k] = t;
                        }
                    }
                }
            }
            float mine = 0.f;   // lane k keeps row r0 + k
#pragma unroll
            for (int k = 0; k < LIN_ROWS; ++k) {
                const float v = warp_sum(acc[k]);
                if (lane == k) mine = v;
            }
            if (KS > 1) {
                if (lane < LIN_ROWS) part[warp][lane] = mine;
                __syncthreads();
                if (slice == 0 && lane < LIN_ROWS) {
                    float t = part[warp][lane];
#pragma unroll
                    for (int sl = 1; sl < KS; ++sl) t += part[warp + sl][lane];
                    mine = t;
                }
                __syncthreads();   // part is reused by the next row group
            }
            const int r = r0 + lane;
            if (slice == 0 && live && lane < LIN_ROWS && r < a.rows) {
                float v = mine + bo;
                if (a.gelu) v = gelu_tanh_f(v);
                if (a.res) v += a.res[(size_t)r * a.ldr + o];
                a.y[(size_t)r * a.ldy + o] = v;
            }
        }
    }
}

// The same product streamed through shared memory, for bf16 weights (16-byte aligned, in a
// multiple of 8 and at most LP_MAX_IN), 16-byte aligned activation rows (ldx a multiple of 4) and
// no head-select: a persistent CTA walks groups of LP_ROWS consecutive output features; their
// weight rows (contiguous) arrive by per-thread 16-byte cp.async copies into a ring of NST
// stages, the first ones issued before the dependency wait (weights do not depend on the previous
// kernel). Thread t takes the 8-column chunks t, t + 256, ... of the inputs for all LP_ROWS
// features of a group, so each chunk of LP_XR activation rows it loads serves all of them (as
// many activation bytes as weight bytes, where one warp per feature read LIN_ROWS activation
// chunks per weight chunk and was bound by those L1 reads); the per-feature sums are reduced over
// the block in a fixed order. No waits that can spin: the copies are waited with
// cp.async.wait_group.
constexpr int LP_ROWS = 8;
constexpr int LP_XR = 4;          // activation rows per pass
constexpr int LP_MAX_IN = 4096;
__host__ __device__ constexpr int lp_stages(int in) {
    return in <= 2048 ? 4 : 3;
}
template <int NST>
__global__ void __launch_bounds__(256) k_corr_linear_pipe(const LinArgs a) {
    extern __shared__ __align__(128) uint8_t lp_smem[];
    __shared__ float red[8][LP_ROWS * LP_XR];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int in = a.in, nch = in / 8;
    const int sbytes = LP_ROWS * in * 2;
    const int ngroups = (a.out + LP_ROWS - 1) / LP_ROWS;
    const uint8_t* W = static_cast<const uint8_t*>(a.w);
    // Group k of this CTA: blockIdx.x + k gridDim.x; its rows into stage k mod NST (one commit
    // group per k, empty past the last group, so the group count stays uniform).
    auto issue = [&](int k) {
        const int g = blockIdx.x + k * gridDim.x;
        if (g < ngroups) {
            const int rows = min(LP_ROWS, a.out - g * LP_ROWS);
            const int chunks = rows * nch;
            const uint8_t* src = W + (size_t)g * LP_ROWS * in * 2;
            const uint32_t dst = jpi::ptx::smem_u32(lp_smem + (size_t)(k % NST) * sbytes);
            for (int c = tid; c < chunks; c += 256) jpi::ptx::cp_async_16(dst + 16 * c, src + 16 * (size_t)c, true);
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
#pragma unroll
    for (int k = 0; k < NST - 1; ++k) issue(k);
    jpi::ptx::grid_dep_wait();
    jpi::ptx::grid_dep_launch();
    for (int k = 0; blockIdx.x + k * gridDim.x < ngroups; ++k) {
        issue(k + NST - 1);
        asm volatile("cp.async.wait_group %0;" ::"n"(NST - 1) : "memory");
        __syncthreads();   // stage k mod NST holds group k for every thread
        const int o0 = (blockIdx.x + k * gridDim.x) * LP_ROWS;
        const int nout = min(LP_ROWS, a.out - o0);
        const uint4* wst = reinterpret_cast<const uint4*>(lp_smem + (size_t)(k % NST) * sbytes);
        for (int r0 = 0; r0 < a.rows; r0 += LP_XR) {
            const int nr = min(LP_XR, a.rows - r0);
            // The bias and residual of this thread's output (thread o LP_XR + q writes feature
            // o0 + o of row r0 + q), fetched before the products so their latency hides there.
            float bias_v = 0.f, res_v = 0.f;
            if (tid < LP_ROWS * LP_XR) {
                const int o = tid / LP_XR, q = tid % LP_XR;
                if (o < nout && q < nr) {
                    if (a.bias) bias_v = a.bias[o0 + o];
                    if (a.res) res_v = a.res[(size_t)(r0 + q) * a.ldr + o0 + o];
                }
            }
            float acc[LP_ROWS][LP_XR];
#pragma unroll
            for (int o = 0; o < LP_ROWS; ++o)
#pragma unroll
                for (int q = 0; q < LP_XR; ++q) acc[o][q] = 0.f;
            for (int c = tid; c < nch; c += 256) {
                float x[LP_XR][8];
#pragma unroll
                for (int q = 0; q < LP_XR; ++q) {
                    float4 x0 = make_float4(0.f, 0.f, 0.f, 0.f), x1 = x0;
                    if (q < nr) {
                        const float* xr = a.x + (size_t)(r0 + q) * a.ldx + 8 * c;
                        x0 = *reinterpret_cast<const float4*>(xr);
                        x1 = *reinterpret_cast<const float4*>(xr + 4);
                    }
                    x[q][0] = x0.x; x[q][1] = x0.y; x[q][2] = x0.z; x[q][3] = x0.w;
                    x[q][4] = x1.x; x[q][5] = x1.y; x[q][6] = x1.z; x[q][7] = x1.w;
                }
#pragma unroll
                for (int o = 0; o < LP_ROWS; ++o) {
                    if (o >= nout) break;
                    const uint4 wv = wst[(size_t)o * nch + c];
                    const uint32_t u[4] = {wv.x, wv.y, wv.z, wv.w};
                    float w[8];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u[e]));
                        w[2 * e] = f.x;
                        w[2 * e + 1] = f.y;
                    }
#pragma unroll
                    for (int q = 0; q < LP_XR; ++q) {
                        float t = acc[o][q];
#pragma unroll
                        for (int e = 0; e < 8; ++e) t = fmaf(w[e], x[q][e], t);
                        acc[o][q] = t;
                    }
                }
            }
            // (feature o, row q) sums: over the warp's lanes, then over the 8 warps in order. The
            // warp sum is a reduce-scatter: at offset 16, 8, .., 1 each lane keeps the half of its
            // pairs whose bit matches its own and adds its partner's partial of them (the same
            // pairwise sums as a butterfly per pair, 31 shuffles instead of 160); lane p ends
            // with pair p = o LP_XR + q.
            static_assert(LP_ROWS * LP_XR == 32, "one pair per lane");
            float pv[32];
#pragma unroll
            for (int o = 0; o < LP_ROWS; ++o)
#pragma unroll
                for (int q = 0; q < LP_XR; ++q) pv[o * LP_XR + q] = acc[o][q];
#pragma unroll
            for (int sh = 16; sh > 0; sh >>= 1) {
                const bool hi = (lane & sh) != 0;
#pragma unroll
                for (int i = 0; i < sh; ++i) {
                    const float send = hi ? pv[i] : pv[i + sh];
                    const float keep = hi ? pv[i + sh] : pv[i];
                    pv[i] = keep + __shfl_xor_sync(0xffffffffu, send, sh);
                }
            }
            red[warp][lane] = pv[0];
            __syncthreads();
            if (tid < LP_ROWS * LP_XR) {
                const int o = tid / LP_XR, q = tid % LP_XR;
                float v = 0.f;
#pragma unroll
                for (int w8 = 0; w8 < 8; ++w8) v += red[w8][tid];
                const int of = o0 + o, r = r0 + q;
                if (o < nout && q < nr) {
                    v += bias_v;
                    if (a.gelu) v = gelu_tanh_f(v);
                    if (a.res) v += res_v;
                    a.y[(size_t)r * a.ldy + of] = v;
                }
            }
            __syncthreads();   // red is reused by the next pass
        }
    }
    asm volatile("cp.async.wait_group 0;" ::: "memory");   // nothing lands after exit
}

// LayerNorm of `rows` rows of width d: one warp per row (grid-stride over rows), three passes
// (mean, biased variance, output). VEC: every row and vector 16-byte aligned, d a multiple of 4,
// so the passes move float4s.
template <bool VEC>
__global__ void __launch_bounds__(256) k_corr_layernorm(const float* __restrict__ x, int ldx,
                                                        const float* __restrict__ g,
                                                        const float* __restrict__ b,
                                                        float* __restrict__ y, int ldy, int rows,
                                                        int d, float eps) {
    // Launched with programmatic dependent launch: wait for the previous kernel's results, then
    // let the next kernel's CTAs be scheduled (they wait in turn).
    jpi::ptx::grid_dep_wait();
    jpi::ptx::grid_dep_launch();
    const int lane = threadIdx.x & 31, nwarps = (int)((gridDim.x * blockDim.x) >> 5);
    for (int r = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5); r < rows; r += nwarps) {
        const float* xr = x + (size_t)r * ldx;
        float* yr = y + (size_t)r * ldy;
        if (VEC) {
            const int d4 = d >> 2;
            const float4* x4 = reinterpret_cast<const float4*>(xr);
            float s = 0.f;
#pragma unroll 8
            for (int i = lane; i < d4; i += 32) {
                const float4 v = x4[i];
                s += (v.x + v.y) + (v.z + v.w);
            }
            const float mean = warp_sum(s) / (float)d;
            float var = 0.f;
#pragma unroll 4
            for (int i = lane; i < d4; i += 32) {
                const float4 v = x4[i];
                const float t0 = v.x - mean, t1 = v.y - mean, t2 = v.z - mean, t3 = v.w - mean;
                var = fmaf(t0, t0, fmaf(t1, t1, fmaf(t2, t2, fmaf(t3, t3, var))));
            }
            const float rstd = 1.f / sqrtf(warp_sum(var) / (float)d + eps);
            float4* y4 = reinterpret_cast<float4*>(yr);
            const float4* g4 = reinterpret_cast<const float4*>(g);
            const float4* b4 = reinterpret_cast<const float4*>(b);
#pragma unroll 4
            for (int i = lane; i < d4; i += 32) {
                const float4 v = x4[i], gg = g4[i], bb = b4[i];
                y4[i] = make_float4((v.x - mean) * rstd * gg.x + bb.x, (v.y - mean) * rstd * gg.y + bb.y,
                                    (v.z - mean) * rstd * gg.z + bb.z, (v.w - mean) * rstd * gg.w + bb.w);
            }
        } else {
            float s = 0.f;
            for (int i = lane; i < d; i += 32) s += xr[i];
            const float mean = warp_sum(s) / (float)d;
            float var = 0.f;
            for (int i = lane; i < d; i += 32) {
                const float t = xr[i] - mean;
                var = fmaf(t, t, var);
            }
            const float rstd = 1.f / sqrtf(warp_sum(var) / (float)d + eps);
            for (int i = lane; i < d; i += 32) yr[i] = (xr[i] - mean) * rstd * g[i] + b[i];
        }
    }
}

// Multi-head attention over few keys: query row (b, i) of head h against key rows (b, j),
// j < nk, every key visible. One warp per (b, h, i); head_dim <= 256, nk <= 64.
struct AttnSmallArgs {
    const float* q;
    int ldq;
    const float* k;
    int ldk;
    const float* v;
    int ldv;
    float* o;
    int ldo;
    int B, nq, nk, H, Dh;
    float scale;
};

__global__ void __launch_bounds__(256) k_corr_attn(const AttnSmallArgs a) {
    // Launched with programmatic dependent launch: wait for the previous kernel's results, then
    // let the next kernel's CTAs be scheduled (they wait in turn).
    jpi::ptx::grid_dep_wait();
    jpi::ptx::grid_dep_launch();
    __shared__ float sp[8][JPI_CORR_MAX_DELTA];
    const int wib = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int gw = blockIdx.x * 8 + wib;
    if (gw >= a.B * a.H * a.nq) return;   // whole warps leave; no block barrier follows
    const int i = gw % a.nq, h = (gw / a.nq) % a.H, b = gw / (a.nq * a.H);
    const float* qr = a.q + (size_t)(b * a.nq + i) * a.ldq + h * a.Dh;
    float qf[8];
#pragma unroll
    for (int t = 0; t < 8; ++t) {
        const int d = lane + 32 * t;
        qf[t] = d < a.Dh ? qr[d] : 0.f;
    }
    // Keys (and below, values) four rows at a time: their loads are in flight together.
    float mx = -INFINITY;
    for (int j0 = 0; j0 < a.nk; j0 += 4) {
        float kv[4][8];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int j = j0 + u < a.nk ? j0 + u : j0;
            const float* kr = a.k + (size_t)(b * a.nk + j) * a.ldk + h * a.Dh;
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                const int d = lane + 32 * t;
                kv[u][t] = d < a.Dh ? kr[d] : 0.f;
            }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int j = j0 + u;
            if (j >= a.nk) break;
            float s = 0.f;
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                const int d = lane + 32 * t;
                if (d < a.Dh) s = fmaf(qf[t], kv[u][t], s);
            }
            s = warp_sum(s) * a.scale;
            if (lane == 0) sp[wib][j] = s;
            mx = fmaxf(mx, s);
        }
    }
    __syncwarp();
    float den = 0.f;
    for (int j = lane; j < a.nk; j += 32) {
        const float e = expf(sp[wib][j] - mx);
        sp[wib][j] = e;
        den += e;
    }
    den = warp_sum(den);
    __syncwarp();
    float of[8];
#pragma unroll
    for (int t = 0; t < 8; ++t) of[t] = 0.f;
    for (int j0 = 0; j0 < a.nk; j0 += 4) {
        float vv[4][8];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int j = j0 + u < a.nk ? j0 + u : j0;
            const float* vr = a.v + (size_t)(b * a.nk + j) * a.ldv + h * a.Dh;
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                const int d = lane + 32 * t;
                vv[u][t] = d < a.Dh ? vr[d] : 0.f;
            }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int j = j0 + u;
            if (j >= a.nk) break;
            const float p = sp[wib][j];
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                const int d = lane + 32 * t;
                if (d < a.Dh) of[t] = fmaf(p, vv[u][t], of[t]);
            }
        }
    }
    const float inv = 1.f / den;
    float* orow = a.o + (size_t)(b * a.nq + i) * a.ldo + h * a.Dh;
#pragma unroll
    for (int t = 0; t < 8; ++t) {
        const int d = lane + 32 * t;
        if (d < a.Dh) orow[d] = of[t] * inv;
    }
}

// Create time: a[h T' + i][c] = scale * sum_e qc[i][h Dh + e] wk[h Dh + e][c] (the cross-
// attention's scaled queries mapped into VLM space). Grid (ceil(dv / 256), H).
template <typename TW>
__global__ void __launch_bounds__(256) k_corr_qk(const float* __restrict__ qc, const TW* __restrict__ wk,
                                                 float* __restrict__ qk, int T, int Dh, int d, int dv,
                                                 float scale) {
    // Launched with programmatic dependent launch: wait for the previous kernel's results, then
    // let the next kernel's CTAs be scheduled (they wait in turn).
    jpi::ptx::grid_dep_wait();
    jpi::ptx::grid_dep_launch();
    __shared__ float qs[JPI_MAX_CORRECTION][256];
    const int h = blockIdx.y, c = blockIdx.x * 256 + threadIdx.x;
    for (int idx = threadIdx.x; idx < T * Dh; idx += 256)
        qs[idx / Dh][idx % Dh] = qc[(size_t)(idx / Dh) * d + h * Dh + idx % Dh];
    __syncthreads();
    if (c >= dv) return;
    float acc[JPI_MAX_CORRECTION];
#pragma unroll
    for (int i = 0; i < JPI_MAX_CORRECTION; ++i) acc[i] = 0.f;
    for (int e = 0; e < Dh; ++e) {
        const float w = to_f(wk[(size_t)(h * Dh + e) * dv + c]);
#pragma unroll
        for (int i = 0; i < JPI_MAX_CORRECTION; ++i)
            if (i < T) acc[i] = fmaf(qs[i][e], w, acc[i]);
    }
#pragma unroll
    for (int i = 0; i < JPI_MAX_CORRECTION; ++i)
        if (i < T) qk[((size_t)h * T + i) * dv + c] = acc[i] * scale;
}

// Partial scores over one chunk of the VLM features: part[b][kc][m][j] = sum over c in chunk kc
// (CORR_KCHUNK features) of qk[m][c] hv[b][j][c], m < M, j < T. Grid (ceil(T / 32), chunks, B):
// 32 tokens per CTA; the chunk's query rows and token rows are staged in shared memory (fp32) with
// all their loads in flight together, then thread (mg, jg) = (tid / 16, tid mod 16) computes the
// register tile of rows mg, mg + 16, .. (< M) x tokens jg, jg + 16 from 16-byte loads of both
// operands (four features at a time, summed in feature order). Splitting the feature sum over
// CTAs keeps the whole GPU busy at batch 1 (26 token tiles alone would not); the chunks are added
// in order by k_corr_softmax_sum.
constexpr int CORR_KCHUNK = 256;
constexpr int CORR_KPAD = CORR_KCHUNK + 4;   // 16-byte rows; 8 consecutive rows hit distinct banks
constexpr size_t CORR_SCORES_SMEM = (size_t)(CORR_MAX_M + 32) * CORR_KPAD * sizeof(float);

// VEC: dv a multiple of 4 and hv aligned to four elements, so the staging moves four features
// per load; every thread's staging loads are issued before any of its stores (one at a time, each
// store would hold the next load back for a full L2 round trip).
template <typename THV, bool VEC>
__global__ void __launch_bounds__(256) k_corr_scores(const float* __restrict__ qk, const THV* __restrict__ hv,
                                                     float* __restrict__ part, int M, int T, int dv) {
    // Launched with programmatic dependent launch: wait for the previous kernel's results, then
    // let the next kernel's CTAs be scheduled (they wait in turn).
    jpi::ptx::grid_dep_wait();
    jpi::ptx::grid_dep_launch();
    extern __shared__ float4 sm_scores4[];
    float* as = reinterpret_cast<float*>(sm_scores4);   // [M][CORR_KPAD]
    float* bs = as + CORR_MAX_M * CORR_KPAD;            // [32][CORR_KPAD]
    const int b = blockIdx.z, kc = blockIdx.y, j0 = blockIdx.x * 32;
    const int c0 = kc * CORR_KCHUNK, cn = min(CORR_KCHUNK, dv - c0);
    const THV* hb = hv + (size_t)b * T * dv;
    if (VEC) {
        // Thread t takes feature quad t mod 64 of rows t / 64, t / 64 + 4, ..: CORR_MAX_M / 4 query
        // rows and 8 token rows at most.
        const int k4 = threadIdx.x & 63, r0 = threadIdx.x >> 6, kk = 4 * k4;
        const bool kin = kk < cn;
        float4 qa[CORR_MAX_M / 4], hb4[8];
#pragma unroll
        for (int i = 0; i < CORR_MAX_M / 4; ++i) {
            const int m = r0 + 4 * i;
            qa[i] = (m < M && kin) ? *reinterpret_cast<const float4*>(qk + (size_t)m * dv + c0 + kk)
                                   : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const int j = j0 + r0 + 4 * i;
            hb4[i] = (j < T && kin) ? load4(hb + (size_t)j * dv + c0 + kk) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int i = 0; i < CORR_MAX_M / 4; ++i) {
            const int m = r0 + 4 * i;
            if (m < M) *reinterpret_cast<float4*>(as + m * CORR_KPAD + kk) = qa[i];
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) *reinterpret_cast<float4*>(bs + (r0 + 4 * i) * CORR_KPAD + kk) = hb4[i];
    } else {
        for (int idx = threadIdx.x; idx < M * CORR_KCHUNK; idx += 256) {
            const int m = idx / CORR_KCHUNK, kk = idx % CORR_KCHUNK;
            as[m * CORR_KPAD + kk] = kk < cn ? qk[(size_t)m * dv + c0 + kk] : 0.f;
        }
        for (int idx = threadIdx.x; idx < 32 * CORR_KCHUNK; idx += 256) {
            const int t = idx / CORR_KCHUNK, kk = idx % CORR_KCHUNK, j = j0 + t;
            bs[t * CORR_KPAD + kk] = (j < T && kk < cn) ? to_f(hb[(size_t)j * dv + c0 + kk]) : 0.f;
        }
    }
    __syncthreads();
    constexpr int RM = CORR_MAX_M / 16;   // rows per thread at most
    const int mg = threadIdx.x >> 4, jg = threadIdx.x & 15;
    float acc[RM][2];
#pragma unroll
    for (int r = 0; r < RM; ++r) acc[r][0] = acc[r][1] = 0.f;
    const float4* b0 = reinterpret_cast<const float4*>(bs + jg * CORR_KPAD);
    const float4* b1 = reinterpret_cast<const float4*>(bs + (jg + 16) * CORR_KPAD);
#pragma unroll 4
    for (int k4 = 0; k4 < CORR_KCHUNK / 4; ++k4) {
        const float4 x0 = b0[k4], x1 = b1[k4];
#pragma unroll
        for (int r = 0; r < RM; ++r) {
            const int m = mg + 16 * r;
            if (m < M) {
                const float4 q = reinterpret_cast<const float4*>(as + m * CORR_KPAD)[k4];
                acc[r][0] = fmaf(q.w, x0.w, fmaf(q.z, x0.z, fmaf(q.y, x0.y, fmaf(q.x, x0.x, acc[r][0]))));
                acc[r][1] = fmaf(q.w, x1.w, fmaf(q.z, x1.z, fmaf(q.y, x1.y, fmaf(q.x, x1.x, acc[r][1]))));
            }
        }
    }
#pragma unroll
    for (int r = 0; r < RM; ++r) {
        const int m = mg + 16 * r;
        if (m >= M) continue;
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int j = j0 + jg + 16 * u;
            if (j < T) part[(((size_t)b * gridDim.y + kc) * M + m) * T + j] = acc[r][u];
        }
    }
}

// Block-wide reductions over 256 threads (8 warps), through `red` [8] in shared memory.
__device__ __forceinline__ float block_max256(float v, float* red) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    float r = red[0];
#pragma unroll
    for (int w = 1; w < 8; ++w) r = fmaxf(r, red[w]);
    __syncthreads();
    return r;
}
__device__ __forceinline__ float block_sum256(float v, float* red) {
    v = warp_sum(v);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    float r = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) r += red[w];   // fixed order
    __syncthreads();
    return r;
}

// Row r = b M + m of the scores (one CTA of 256 threads per row): the nkc feature chunks added in
// order, then the softmax over its n tokens, written to s[r][.].
__global__ void __launch_bounds__(256) k_corr_softmax_sum(const float* __restrict__ part, float* __restrict__ s,
                                                          int M, int n, int nkc) {
    // Launched with programmatic dependent launch: wait for the previous kernel's results, then
    // let the next kernel's CTAs be scheduled (they wait in turn).
    jpi::ptx::grid_dep_wait();
    jpi::ptx::grid_dep_launch();
    __shared__ float red[8];
    const int r = blockIdx.x, b = r / M, m = r - b * M;
    const float* p0 = part + ((size_t)b * nkc * M + m) * n;
    float* row = s + (size_t)r * n;
    float mx = -INFINITY;
    for (int j = threadIdx.x; j < n; j += 256) {
        float v = 0.f;
        for (int kc = 0; kc < nkc; ++kc) v += p0[(size_t)kc * M * n + j];
        row[j] = v;
        mx = fmaxf(mx, v);
    }
    mx = block_max256(mx, red);
    float den = 0.f;
    for (int j = threadIdx.x; j < n; j += 256) {
        const float e = expf(row[j] - mx);
        row[j] = e;
        den += e;
    }
    const float inv = 1.f / block_sum256(den, red);
    for (int j = threadIdx.x; j < n; j += 256) row[j] *= inv;
}

// Partial weighted sums over one chunk of CORR_TCHUNK tokens: part[b][tc][m][c] = sum over j in
// chunk tc of p[b][m][j] hv[b][j][c]. Grid (ceil(dv / 256), chunks, B): thread (cg, mg) =
// (tid mod 128, tid / 128) takes columns 2 cg, 2 cg + 1 of the CTA's 256 and rows mg RH .. + RH - 1
// (RH = 16 for M <= 32, else 32), token after token in order; the chunk's probabilities sit in
// shared memory transposed ([token][row], read as 16-byte broadcasts) and each token's two values
// come in one load, eight tokens' loads in flight together. The token chunks are added in order
// by k_corr_wsum_reduce.
constexpr int CORR_TCHUNK = 64;
constexpr int CORR_PTS = CORR_MAX_M + 4;   // row stride of the transposed probabilities

template <typename THV>
__device__ __forceinline__ float2 load2(const THV* p);
template <>
__device__ __forceinline__ float2 load2<float>(const float* p) { return __ldg(reinterpret_cast<const float2*>(p)); }
template <>
__device__ __forceinline__ float2 load2<__nv_bfloat16>(const __nv_bfloat16* p) {
    const uint32_t u = __ldg(reinterpret_cast<const unsigned int*>(p));
    return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u));
}

// PAIR: dv even and hv aligned to two elements, so a thread's two columns load together; else
// each value on its own (and a last odd column alone).
template <typename THV, int RH, bool PAIR>
__global__ void __launch_bounds__(256) k_corr_wsum(const float* __restrict__ p, const THV* __restrict__ hv,
                                                   float* __restrict__ part, int M, int T, int dv) {
    // Launched with programmatic dependent launch: wait for the previous kernel's results, then
    // let the next kernel's CTAs be scheduled (they wait in turn).
    jpi::ptx::grid_dep_wait();
    jpi::ptx::grid_dep_launch();
    __shared__ __align__(16) float pt[CORR_TCHUNK][CORR_PTS];
    const int b = blockIdx.z, tc = blockIdx.y;
    const int j0 = tc * CORR_TCHUNK, jn = min(CORR_TCHUNK, T - j0);
    {
        // Thread t loads token t mod 64 of rows t / 64, t / 64 + 4, .. (coalesced along the
        // tokens, all loads before the transposed stores); rows past M are zero.
        const int jj = threadIdx.x & 63, r0 = threadIdx.x >> 6;
        float pv[CORR_PTS / 4];
#pragma unroll
        for (int i = 0; i < CORR_PTS / 4; ++i) {
            const int r = r0 + 4 * i;
            pv[i] = (jj < jn && r < M) ? p[((size_t)b * M + r) * T + j0 + jj] : 0.f;
        }
#pragma unroll
        for (int i = 0; i < CORR_PTS / 4; ++i) pt[jj][r0 + 4 * i] = pv[i];
    }
    __syncthreads();
    const int cg = threadIdx.x & 127, mg = threadIdx.x >> 7;
    const int c = blockIdx.x * 256 + 2 * cg;
    if (c >= dv) return;
    const int m0 = mg * RH;
    float acc[RH][2];
#pragma unroll
    for (int i = 0; i < RH; ++i) acc[i][0] = acc[i][1] = 0.f;
    const THV* hb = hv + ((size_t)b * T + j0) * dv + c;
    for (int jb = 0; jb < jn; jb += 8) {
        float2 hvv[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            hvv[u] = make_float2(0.f, 0.f);
            if (jb + u < jn) {
                const THV* hp = hb + (size_t)(jb + u) * dv;
                if (PAIR) hvv[u] = load2(hp);
                else hvv[u] = make_float2(load1(hp), c + 1 < dv ? load1(hp + 1) : 0.f);
            }
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const float4* prow = reinterpret_cast<const float4*>(&pt[jb + u][m0]);
#pragma unroll
            for (int i4 = 0; i4 < RH / 4; ++i4) {
                const float4 pw = prow[i4];
                const float w4[4] = {pw.x, pw.y, pw.z, pw.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    acc[4 * i4 + e][0] = fmaf(w4[e], hvv[u].x, acc[4 * i4 + e][0]);
                    acc[4 * i4 + e][1] = fmaf(w4[e], hvv[u].y, acc[4 * i4 + e][1]);
                }
            }
        }
    }
    float* out = part + ((size_t)b * gridDim.y + tc) * M * dv + c;
#pragma unroll
    for (int i = 0; i < RH; ++i) {
        const int m = m0 + i;
        if (m >= M) continue;
        if (PAIR) {
            *reinterpret_cast<float2*>(out + (size_t)m * dv) = make_float2(acc[i][0], acc[i][1]);
        } else {
            out[(size_t)m * dv] = acc[i][0];
            if (c + 1 < dv) out[(size_t)m * dv + 1] = acc[i][1];
        }
    }
}

// g[b][m][c] = the ntc token-chunk partials added in order.
__global__ void k_corr_wsum_reduce(const float* __restrict__ part, float* __restrict__ g, int B, int M, int dv,
                                   int ntc) {
    // Launched with programmatic dependent launch: wait for the previous kernel's results, then
    // let the next kernel's CTAs be scheduled (they wait in turn).
    jpi::ptx::grid_dep_wait();
    jpi::ptx::grid_dep_launch();
    const long long total = (long long)B * M * dv;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x) {
        const long long b = idx / ((long long)M * dv), rest = idx - b * M * dv;
        const float* p0 = part + (size_t)b * ntc * M * dv + rest;
        float v = 0.f;
        for (int tc = 0; tc < ntc; ++tc) v += p0[(size_t)tc * M * dv];
        g[idx] = v;
    }
}

// y[(b n + k)][c] += pos[k][c] for b < B, k < n, c < d.
__global__ void k_corr_add_pos(float* __restrict__ y, const float* __restrict__ pos, int B, int n, int d) {
    // Launched with programmatic dependent launch: wait for the previous kernel's results, then
    // let the next kernel's CTAs be scheduled (they wait in turn).
    jpi::ptx::grid_dep_wait();
    jpi::ptx::grid_dep_launch();
    const long long total = (long long)B * n * d;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x) {
        const int c = (int)(idx % d);
        const int k = (int)((idx / d) % n);
        y[idx] += pos[(size_t)k * d + c];
    }
}

// xj[(b T' + i)][0 .. d) = state[b][i][.], xj[(b T' + i)][d .. 2d) = summary[b][.].
__global__ void k_corr_join(const float* __restrict__ state, const float* __restrict__ summary,
                            float* __restrict__ xj, int B, int T, int d) {
    // Launched with programmatic dependent launch: wait for the previous kernel's results, then
    // let the next kernel's CTAs be scheduled (they wait in turn).
    jpi::ptx::grid_dep_wait();
    jpi::ptx::grid_dep_launch();
    const long long total = (long long)B * T * 2 * d;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x) {
        const int c = (int)(idx % (2 * d));
        const long long r = idx / (2 * d);   // b T' + i
        const int b = (int)(r / T);
        xj[idx] = c < d ? state[r * d + c] : summary[(size_t)b * d + (c - d)];
    }
}

// conf[b] = w . mean_i u[b T' + i] + bias; one CTA of 256 threads per request.
__global__ void __launch_bounds__(256) k_corr_confidence(const float* __restrict__ u, const float* __restrict__ w,
                                                         const float* __restrict__ bias, float* __restrict__ conf,
                                                         int T, int d) {
    // Launched with programmatic dependent launch: wait for the previous kernel's results, then
    // let the next kernel's CTAs be scheduled (they wait in turn).
    jpi::ptx::grid_dep_wait();
    jpi::ptx::grid_dep_launch();
    __shared__ float red[8];
    const int b = blockIdx.x;
    float s = 0.f;
    for (int c = threadIdx.x; c < d; c += 256) {
        float m = 0.f;
        for (int i = 0; i < T; ++i) m += u[((size_t)b * T + i) * d + c];
        s = fmaf(w[c], m / (float)T, s);
    }
    s = block_sum256(s, red);
    if (threadIdx.x == 0) conf[b] = s + bias[0];
}

__global__ void k_corr_cast(const float* __restrict__ src, __nv_bfloat16* __restrict__ dst, long long n) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
         i += (long long)gridDim.x * blockDim.x)
        dst[i] = __float2bfloat16_rn(src[i]);
}

// dst[r n + i] = src[i] for r < reps, i < n. src may be the start of dst: the first n elements are
// rewritten with their own values.
__global__ void k_corr_repeat(const float* src, float* dst, long long n, int reps) {
    // Launched with programmatic dependent launch: wait for the previous kernel's results, then
    // let the next kernel's CTAs be scheduled (they wait in turn).
    jpi::ptx::grid_dep_wait();
    jpi::ptx::grid_dep_launch();
    const long long total = n * reps;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x)
        dst[i] = src[i % n];
}

int grid_for(long long threads, int block = 256, int cap = 8192) {
    long long g = (threads + block - 1) / block;
    if (g < 1) g = 1;
    if (g > cap) g = cap;
    return (int)g;
}

// Device copy of one block: q/k/v rows packed as [wq; wk; wv] ([3d][d]) with [bq; bk; bv].
struct BlockDev {
    float *ln1_w = nullptr, *ln1_b = nullptr;
    void* wqkv = nullptr;
    float* bqkv = nullptr;
    void* wo = nullptr;
    float* bo = nullptr;
    float *ln2_w = nullptr, *ln2_b = nullptr;
    void* w1 = nullptr;
    float* b1 = nullptr;
    void* w2 = nullptr;
    float* b2 = nullptr;
};

}  // namespace

struct jpi_corr_handle {
    jpi_corr_config cfg;
    bool bf16 = true;
    int num_sms = 0;   // persistent CTAs of the streamed products
    int d = 0, H = 0, Dh = 0, F = 0, dv = 0, Ti = 0, A = 0, Dm = 0, J = 0, B = 0, Tm = 0, M = 0;
    std::vector<void*> allocs;
    size_t bytes = 0;
    float* staging = nullptr;   // fp32 device staging for host weights
    size_t staging_elems = 0;

    // Weights.
    float* qf_query = nullptr;   // [T'][d]
    BlockDev qf_sa;
    float *qf_ln2_w = nullptr, *qf_ln2_b = nullptr;
    void *qf_ca_wq = nullptr, *qf_ca_wk = nullptr, *qf_ca_wv = nullptr, *qf_ca_wo = nullptr;
    float *qf_ca_bq = nullptr, *qf_ca_bv = nullptr, *qf_ca_bo = nullptr;
    float *qf_ln3_w = nullptr, *qf_ln3_b = nullptr, *qf_lnf_w = nullptr, *qf_lnf_b = nullptr;
    void *qf_w1 = nullptr, *qf_w2 = nullptr;
    float *qf_b1 = nullptr, *qf_b2 = nullptr;
    void *act_w1 = nullptr, *act_w2 = nullptr;
    float *act_b1 = nullptr, *act_b2 = nullptr, *act_pos = nullptr;
    BlockDev ab;
    void* fuse_w = nullptr;
    float* fuse_b = nullptr;
    std::vector<BlockDev> jb;
    float *head_ln_w = nullptr, *head_ln_b = nullptr;
    void* corr_w = nullptr;
    float *corr_b = nullptr, *conf_w = nullptr, *conf_b = nullptr;

    // Weight-only values computed at create time.
    float* x1b = nullptr;   // [B T'][d] the queries after their self-attention, per request slot
    float* qk = nullptr;    // [H T'][dv] cross-attention queries mapped into VLM space (scaled)

    // Activations (fp32).
    float *t1 = nullptr, *xa = nullptr, *ua = nullptr, *kva = nullptr;   // [B Dm][d], kva [B Dm][2d]
    float *ql = nullptr, *ol = nullptr, *xl = nullptr, *ul = nullptr;    // [B][d]
    float* hidl = nullptr;                                                // [B][F]
    float *xj = nullptr, *xf = nullptr, *u = nullptr, *qkv = nullptr, *o = nullptr;   // [B T'] rows
    float* hid = nullptr;                                                 // [B T'][F]
    float *sc = nullptr, *gs = nullptr;                                   // [B][M][Tm], [B][M][dv]
    float *scp = nullptr, *gsp = nullptr;   // partials: [B][dv / 256][M][Tm], [B][Tm / 64][M][dv]
    float* conf_scratch = nullptr;                                        // [B]

    // Graph replay: the calls copy their inputs into these buffers, replay the kernel sequence
    // captured once per (call, batch, tokens or delta, input type), and copy the outputs out.
    void* in_vlm = nullptr;                                               // [B][Tm][dv], fp32 or bf16
    float *in_state = nullptr, *in_act = nullptr;                         // [B T'][d], [B Dm][A]
    float *out_st = nullptr, *out_conf = nullptr;                         // [B T'][d], [B]
    cudaStream_t cap = nullptr;
    std::map<std::tuple<int, int, int, int>, cudaGraphExec_t> graphs;
};

namespace {

template <typename T>
jpi_status corr_alloc(jpi_corr_handle* h, T** p, size_t count) {
    void* q = nullptr;
    const size_t bytes = count * sizeof(T);
    const cudaError_t e = cudaMalloc(&q, bytes ? bytes : 16);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return cfail(JPI_ERR_OOM, "cudaMalloc(%zu bytes) failed: %s", bytes, cudaGetErrorString(e));
    }
    h->allocs.push_back(q);
    h->bytes += bytes;
    *p = static_cast<T*>(q);
    return JPI_OK;
}

// Copies an fp32 tensor of n elements (host or device) to dst: fp32 as is, or rounded to bf16.
jpi_status put(jpi_corr_handle* h, bool on_device, void* dst, bool to_bf16, const float* src, size_t n,
               const char* name) {
    if (!src) return cfail(JPI_ERR_INVALID_ARG, "weight tensor %s is NULL", name);
    const float* dsrc = src;
    if (!on_device) {
        if (!to_bf16) {
            JPI_CUDA_TRY(cudaMemcpy(dst, src, n * sizeof(float), cudaMemcpyHostToDevice));
            return JPI_OK;
        }
        JPI_CUDA_TRY(cudaMemcpy(h->staging, src, n * sizeof(float), cudaMemcpyHostToDevice));
        dsrc = h->staging;
    }
    if (to_bf16) {
        k_corr_cast<<<grid_for((long long)n), 256>>>(dsrc, static_cast<__nv_bfloat16*>(dst), (long long)n);
        JPI_CUDA_TRY(cudaGetLastError());
    } else {
        JPI_CUDA_TRY(cudaMemcpy(dst, dsrc, n * sizeof(float), cudaMemcpyDeviceToDevice));
    }
    return JPI_OK;
}

// A weight matrix (stored bf16 or fp32) and a vector (fp32) of the handle.
jpi_status put_mat(jpi_corr_handle* h, bool dev, void** dst, const float* src, size_t n, const char* name) {
    if (h->bf16) {
        __nv_bfloat16* p = nullptr;
        JPI_TRY(corr_alloc(h, &p, n));
        *dst = p;
    } else {
        float* p = nullptr;
        JPI_TRY(corr_alloc(h, &p, n));
        *dst = p;
    }
    return put(h, dev, *dst, h->bf16, src, n, name);
}

jpi_status put_vec(jpi_corr_handle* h, bool dev, float** dst, const float* src, size_t n, const char* name) {
    JPI_TRY(corr_alloc(h, dst, n));
    return put(h, dev, *dst, false, src, n, name);
}

size_t tw_bytes(const jpi_corr_handle* h) { return h->bf16 ? 2 : 4; }
const void* tw_rows(const jpi_corr_handle* h, const void* base, size_t row, size_t in) {
    return static_cast<const char*>(base) + row * in * tw_bytes(h);
}

jpi_status put_block(jpi_corr_handle* h, bool dev, BlockDev* out, const jpi_corr_block& b, bool with_mlp,
                     const char* name) {
    const size_t d = (size_t)h->d, F = (size_t)h->F;
    char nm[64];
    auto N = [&](const char* f) {
        snprintf(nm, sizeof(nm), "%s.%s", name, f);
        return nm;
    };
    JPI_TRY(put_vec(h, dev, &out->ln1_w, b.ln1_w, d, N("ln1_w")));
    JPI_TRY(put_vec(h, dev, &out->ln1_b, b.ln1_b, d, N("ln1_b")));
    if (h->bf16) {
        __nv_bfloat16* p = nullptr;
        JPI_TRY(corr_alloc(h, &p, 3 * d * d));
        out->wqkv = p;
    } else {
        float* p = nullptr;
        JPI_TRY(corr_alloc(h, &p, 3 * d * d));
        out->wqkv = p;
    }
    char* wq = static_cast<char*>(out->wqkv);
    JPI_TRY(put(h, dev, wq, h->bf16, b.wq, d * d, N("wq")));
    JPI_TRY(put(h, dev, wq + d * d * tw_bytes(h), h->bf16, b.wk, d * d, N("wk")));
    JPI_TRY(put(h, dev, wq + 2 * d * d * tw_bytes(h), h->bf16, b.wv, d * d, N("wv")));
    JPI_TRY(corr_alloc(h, &out->bqkv, 3 * d));
    JPI_TRY(put(h, dev, out->bqkv, false, b.bq, d, N("bq")));
    JPI_TRY(put(h, dev, out->bqkv + d, false, b.bk, d, N("bk")));
    JPI_TRY(put(h, dev, out->bqkv + 2 * d, false, b.bv, d, N("bv")));
    JPI_TRY(put_mat(h, dev, &out->wo, b.wo, d * d, N("wo")));
    JPI_TRY(put_vec(h, dev, &out->bo, b.bo, d, N("bo")));
    if (with_mlp) {
        JPI_TRY(put_vec(h, dev, &out->ln2_w, b.ln2_w, d, N("ln2_w")));
        JPI_TRY(put_vec(h, dev, &out->ln2_b, b.ln2_b, d, N("ln2_b")));
        JPI_TRY(put_mat(h, dev, &out->w1, b.w1, F * d, N("w1")));
        JPI_TRY(put_vec(h, dev, &out->b1, b.b1, F, N("b1")));
        JPI_TRY(put_mat(h, dev, &out->w2, b.w2, d * F, N("w2")));
        JPI_TRY(put_vec(h, dev, &out->b2, b.b2, d, N("b2")));
    }
    return JPI_OK;
}

// ---------------------------------------------------------------- launchers

// Every kernel of a call is launched with programmatic dependent launch (each waits for its
// predecessor at its start), so in the captured graph a kernel's launch overlaps the previous
// kernel's tail. A failed launch leaves its error for the cudaGetLastError check that follows.
template <typename... KArgs, typename... Args>
void pdl(cudaStream_t st, dim3 grid, dim3 block, size_t smem, void (*k)(KArgs...), Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at;
    at.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at.val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = &at;
    cfg.numAttrs = 1;
    (void)cudaLaunchKernelEx(&cfg, k, std::forward<Args>(args)...);
}

jpi_status linear(const jpi_corr_handle* h, cudaStream_t st, const float* x, int ldx, const void* w,
                  const float* bias, const float* res, int ldr, float* y, int ldy, int rows, int in,
                  int out, bool gelu, int hs_items = 0) {
    if (rows <= 0 || out <= 0) return JPI_OK;
    LinArgs a;
    a.x = x;
    a.ldx = ldx;
    a.w = w;
    a.bias = bias;
    a.res = res;
    a.ldr = ldr;
    a.y = y;
    a.ldy = ldy;
    a.rows = rows;
    a.in = in;
    a.out = out;
    a.gelu = gelu ? 1 : 0;
    a.hs_items = hs_items;
    a.hs_heads = h->H;
    a.hs_dh = h->Dh;
    const bool vec = in % 4 == 0 && ldx % 4 == 0 && ((uintptr_t)x & 15) == 0 &&
                     ((uintptr_t)w & (h->bf16 ? 7 : 15)) == 0;
    // bf16 rows of 16-byte chunks up to LP_MAX_IN, no head-select: streamed through shared memory
    // by persistent CTAs, one per SM at most.
    if (h->bf16 && hs_items == 0 && in % 8 == 0 && in <= LP_MAX_IN && ldx % 4 == 0 && ((uintptr_t)x & 15) == 0 &&
        ((uintptr_t)w & 15) == 0) {
        const int groups = (out + LP_ROWS - 1) / LP_ROWS;
        const int nb = groups < h->num_sms ? groups : h->num_sms;
        const int nst = lp_stages(in);
        const size_t smem = (size_t)nst * LP_ROWS * in * 2;
        if (nst == 4) pdl(st, dim3(nb), dim3(256), smem, k_corr_linear_pipe<4>, a);
        else pdl(st, dim3(nb), dim3(256), smem, k_corr_linear_pipe<3>, a);
        JPI_CUDA_TRY(cudaGetLastError());
        return JPI_OK;
    }
    // Other bf16 rows of 16-byte chunks: the streaming kernel, with 2 or 4 warps per output
    // feature while that keeps at least 256 inputs a warp and brings the launch towards 2048 warps.
    if (h->bf16 && in % 8 == 0 && ldx % 4 == 0 && ((uintptr_t)x & 15) == 0 && ((uintptr_t)w & 15) == 0) {
        int ks = 1;
        while (ks < 4 && (long long)out * ks < 2048 && in % (16 * ks) == 0 && in / (2 * ks) >= 256) ks *= 2;
        const int groups = (out + 8 / ks - 1) / (8 / ks);
        const int nb = groups < 4096 ? groups : 4096;
        if (ks == 4) pdl(st, dim3(nb), dim3(256), 0, k_corr_linear16<4>, a);
        else if (ks == 2) pdl(st, dim3(nb), dim3(256), 0, k_corr_linear16<2>, a);
        else pdl(st, dim3(nb), dim3(256), 0, k_corr_linear16<1>, a);
        JPI_CUDA_TRY(cudaGetLastError());
        return JPI_OK;
    }
    const int blocks = grid_for((long long)out * 32, 256, 4096);
    if (h->bf16) {
        if (vec) pdl(st, dim3(blocks), dim3(256), 0, k_corr_linear<__nv_bfloat16, true>, a);
        else pdl(st, dim3(blocks), dim3(256), 0, k_corr_linear<__nv_bfloat16, false>, a);
    } else {
        if (vec) pdl(st, dim3(blocks), dim3(256), 0, k_corr_linear<float, true>, a);
        else pdl(st, dim3(blocks), dim3(256), 0, k_corr_linear<float, false>, a);
    }
    JPI_CUDA_TRY(cudaGetLastError());
    return JPI_OK;
}

jpi_status layernorm(const jpi_corr_handle* h, cudaStream_t st, const float* x, int ldx, const float* g,
                     const float* b, float* y, int ldy, int rows) {
    if (rows <= 0) return JPI_OK;
    const bool vec = h->d % 4 == 0 && ldx % 4 == 0 && ldy % 4 == 0 &&
                     (((uintptr_t)x | (uintptr_t)y | (uintptr_t)g | (uintptr_t)b) & 15) == 0;
    if (vec)
        pdl(st, dim3(grid_for((long long)rows * 32)), dim3(256), 0, k_corr_layernorm<true>, x, ldx, g, b, y, ldy, rows, h->d,
                                                                           h->cfg.ln_eps);
    else
        pdl(st, dim3(grid_for((long long)rows * 32)), dim3(256), 0, k_corr_layernorm<false>, x, ldx, g, b, y, ldy, rows, h->d,
                                                                            h->cfg.ln_eps);
    JPI_CUDA_TRY(cudaGetLastError());
    return JPI_OK;
}

jpi_status attention(const jpi_corr_handle* h, cudaStream_t st, const float* q, int ldq, const float* k,
                     int ldk, const float* v, int ldv, float* o, int ldo, int B, int nq, int nk) {
    AttnSmallArgs a;
    a.q = q;
    a.ldq = ldq;
    a.k = k;
    a.ldk = ldk;
    a.v = v;
    a.ldv = ldv;
    a.o = o;
    a.ldo = ldo;
    a.B = B;
    a.nq = nq;
    a.nk = nk;
    a.H = h->H;
    a.Dh = h->Dh;
    a.scale = 1.f / sqrtf((float)h->Dh);
    const long long warps = (long long)B * h->H * nq;
    pdl(st, dim3((int)((warps + 7) / 8)), dim3(256), 0, k_corr_attn, a);
    JPI_CUDA_TRY(cudaGetLastError());
    return JPI_OK;
}

// One pre-LN block over `rows` rows of x (rows = B n, n tokens per request), in place.
jpi_status block(const jpi_corr_handle* h, cudaStream_t st, const BlockDev& w, float* x, int B, int n) {
    const int d = h->d, rows = B * n;
    JPI_TRY(layernorm(h, st, x, d, w.ln1_w, w.ln1_b, h->u, d, rows));
    JPI_TRY(linear(h, st, h->u, d, w.wqkv, w.bqkv, nullptr, 0, h->qkv, 3 * d, rows, d, 3 * d, false));
    JPI_TRY(attention(h, st, h->qkv, 3 * d, h->qkv + d, 3 * d, h->qkv + 2 * d, 3 * d, h->o, d, B, n, n));
    JPI_TRY(linear(h, st, h->o, d, w.wo, w.bo, x, d, x, d, rows, d, d, false));
    JPI_TRY(layernorm(h, st, x, d, w.ln2_w, w.ln2_b, h->u, d, rows));
    JPI_TRY(linear(h, st, h->u, d, w.w1, w.b1, nullptr, 0, h->hid, h->F, rows, d, h->F, true));
    JPI_TRY(linear(h, st, h->hid, h->F, w.w2, w.b2, x, d, x, d, rows, h->F, d, false));
    return JPI_OK;
}

// Weight-only part of the compressor: x1 = q0 + SA(LN1 q0) for the learned queries q0 (one copy
// per request slot), and the cross-attention queries of LN2 x1 mapped into VLM space.
jpi_status prepare(jpi_corr_handle* h, cudaStream_t st) {
    const int d = h->d, T = h->Ti;
    const BlockDev& sa = h->qf_sa;
    JPI_TRY(layernorm(h, st, h->qf_query, d, sa.ln1_w, sa.ln1_b, h->u, d, T));
    JPI_TRY(linear(h, st, h->u, d, sa.wqkv, sa.bqkv, nullptr, 0, h->qkv, 3 * d, T, d, 3 * d, false));
    JPI_TRY(attention(h, st, h->qkv, 3 * d, h->qkv + d, 3 * d, h->qkv + 2 * d, 3 * d, h->o, d, 1, T, T));
    JPI_TRY(linear(h, st, h->o, d, sa.wo, sa.bo, h->qf_query, d, h->x1b, d, T, d, d, false));
    JPI_TRY(layernorm(h, st, h->x1b, d, h->qf_ln2_w, h->qf_ln2_b, h->u, d, T));
    JPI_TRY(linear(h, st, h->u, d, h->qf_ca_wq, h->qf_ca_bq, nullptr, 0, h->o, d, T, d, d, false));
    const dim3 grid((unsigned)((h->dv + 255) / 256), (unsigned)h->H);
    const float scale = 1.f / sqrtf((float)h->Dh);
    if (h->bf16)
        pdl(st, dim3(grid), dim3(256), 0, k_corr_qk<__nv_bfloat16>, h->o, static_cast<const __nv_bfloat16*>(h->qf_ca_wk),
                                                        h->qk, T, h->Dh, d, h->dv, scale);
    else
        pdl(st, dim3(grid), dim3(256), 0, k_corr_qk<float>, h->o, static_cast<const float*>(h->qf_ca_wk), h->qk, T, h->Dh,
                                               d, h->dv, scale);
    JPI_CUDA_TRY(cudaGetLastError());
    const long long n = (long long)T * d;
    pdl(st, dim3(grid_for(n * h->B)), dim3(256), 0, k_corr_repeat, h->x1b, h->x1b, n, h->B);
    JPI_CUDA_TRY(cudaGetLastError());
    return JPI_OK;
}

jpi_status check_corr_config(const jpi_corr_config* c) {
    if (c->width < 32 || c->width % 32 || c->width > 16384)
        return cfail(JPI_ERR_INVALID_ARG, "width must be a multiple of 32 in [32, 16384]");
    if (c->head_dim < 32 || c->head_dim % 32 || c->head_dim > 256)
        return cfail(JPI_ERR_UNSUPPORTED, "head_dim must be a multiple of 32 and at most 256");
    if (c->n_heads < 1 || c->n_heads * c->head_dim != c->width)
        return cfail(JPI_ERR_INVALID_ARG, "n_heads * head_dim must equal width");
    if (c->mlp_dim < 1 || c->d_vlm < 1 || c->action_dim < 1)
        return cfail(JPI_ERR_INVALID_ARG, "mlp_dim, d_vlm and action_dim must be >= 1");
    if (c->n_items < 1 || c->n_items > JPI_MAX_CORRECTION)
        return cfail(JPI_ERR_UNSUPPORTED, "n_items must be in [1, %d]", JPI_MAX_CORRECTION);
    if (c->n_heads * c->n_items > CORR_MAX_M)
        return cfail(JPI_ERR_UNSUPPORTED, "n_heads * n_items must be at most %d", CORR_MAX_M);
    if (c->max_delta < 1 || c->max_delta > JPI_CORR_MAX_DELTA)
        return cfail(JPI_ERR_UNSUPPORTED, "max_delta must be in [1, %d]", JPI_CORR_MAX_DELTA);
    if (c->n_joint < 0 || c->n_joint > 8) return cfail(JPI_ERR_UNSUPPORTED, "n_joint must be in [0, 8]");
    if (c->max_batch < 1 || c->max_batch > 65535 || c->max_vlm_tokens < 1)
        return cfail(JPI_ERR_INVALID_ARG, "max_batch must be in [1, 65535] and max_vlm_tokens >= 1");
    if ((long long)c->max_batch * c->n_heads * c->n_items * c->max_vlm_tokens > (1ll << 31))
        return cfail(JPI_ERR_UNSUPPORTED, "max_batch * n_heads * n_items * max_vlm_tokens is too large");
    if (c->precision != JPI_BF16 && c->precision != JPI_FP32)
        return cfail(JPI_ERR_INVALID_ARG, "unknown precision %d", (int)c->precision);
    if (!(c->ln_eps >= 0.f)) return cfail(JPI_ERR_INVALID_ARG, "ln_eps must be >= 0");
    return JPI_OK;
}

jpi_status setup(jpi_corr_handle* h, const jpi_corr_config* c, const jpi_corr_weights* w) {
    h->cfg = *c;
    h->bf16 = c->precision == JPI_BF16;
    h->d = c->width;
    h->H = c->n_heads;
    h->Dh = c->head_dim;
    h->F = c->mlp_dim;
    h->dv = c->d_vlm;
    h->Ti = c->n_items;
    h->A = c->action_dim;
    h->Dm = c->max_delta;
    h->J = c->n_joint;
    h->B = c->max_batch;
    h->Tm = c->max_vlm_tokens;
    h->M = h->H * h->Ti;
    const size_t d = (size_t)h->d, F = (size_t)h->F, dv = (size_t)h->dv, T = (size_t)h->Ti;
    const size_t B = (size_t)h->B, Dm = (size_t)h->Dm, A = (size_t)h->A, M = (size_t)h->M;
    const bool dev = w->on_device != 0;
    if (!dev) {
        size_t m = d * d;
        for (size_t v : {F * d, d * dv, Dm * d, 2 * d * d, T * d, d * A}) m = v > m ? v : m;
        JPI_TRY(corr_alloc(h, &h->staging, m));
        h->staging_elems = m;
    }

    // Q-Former compressor.
    JPI_TRY(put_vec(h, dev, &h->qf_query, w->qf_query, T * d, "qf_query"));
    JPI_TRY(put_block(h, dev, &h->qf_sa, w->qf_sa, false, "qf_sa"));
    JPI_TRY(put_vec(h, dev, &h->qf_ln2_w, w->qf_ln2_w, d, "qf_ln2_w"));
    JPI_TRY(put_vec(h, dev, &h->qf_ln2_b, w->qf_ln2_b, d, "qf_ln2_b"));
    JPI_TRY(put_mat(h, dev, &h->qf_ca_wq, w->qf_ca_wq, d * d, "qf_ca_wq"));
    JPI_TRY(put_vec(h, dev, &h->qf_ca_bq, w->qf_ca_bq, d, "qf_ca_bq"));
    JPI_TRY(put_mat(h, dev, &h->qf_ca_wk, w->qf_ca_wk, d * dv, "qf_ca_wk"));
    // qf_ca_bk adds the same amount to every score of a query; softmax cancels it.
    JPI_TRY(put_mat(h, dev, &h->qf_ca_wv, w->qf_ca_wv, d * dv, "qf_ca_wv"));
    JPI_TRY(put_vec(h, dev, &h->qf_ca_bv, w->qf_ca_bv, d, "qf_ca_bv"));
    JPI_TRY(put_mat(h, dev, &h->qf_ca_wo, w->qf_ca_wo, d * d, "qf_ca_wo"));
    JPI_TRY(put_vec(h, dev, &h->qf_ca_bo, w->qf_ca_bo, d, "qf_ca_bo"));
    JPI_TRY(put_vec(h, dev, &h->qf_ln3_w, w->qf_ln3_w, d, "qf_ln3_w"));
    JPI_TRY(put_vec(h, dev, &h->qf_ln3_b, w->qf_ln3_b, d, "qf_ln3_b"));
    JPI_TRY(put_mat(h, dev, &h->qf_w1, w->qf_mlp_w1, F * d, "qf_mlp_w1"));
    JPI_TRY(put_vec(h, dev, &h->qf_b1, w->qf_mlp_b1, F, "qf_mlp_b1"));
    JPI_TRY(put_mat(h, dev, &h->qf_w2, w->qf_mlp_w2, d * F, "qf_mlp_w2"));
    JPI_TRY(put_vec(h, dev, &h->qf_b2, w->qf_mlp_b2, d, "qf_mlp_b2"));
    JPI_TRY(put_vec(h, dev, &h->qf_lnf_w, w->qf_lnf_w, d, "qf_lnf_w"));
    JPI_TRY(put_vec(h, dev, &h->qf_lnf_b, w->qf_lnf_b, d, "qf_lnf_b"));
    // Action branch, join, joint blocks, heads.
    JPI_TRY(put_mat(h, dev, &h->act_w1, w->act_w1, d * A, "act_w1"));
    JPI_TRY(put_vec(h, dev, &h->act_b1, w->act_b1, d, "act_b1"));
    JPI_TRY(put_mat(h, dev, &h->act_w2, w->act_w2, d * d, "act_w2"));
    JPI_TRY(put_vec(h, dev, &h->act_b2, w->act_b2, d, "act_b2"));
    JPI_TRY(put_vec(h, dev, &h->act_pos, w->act_pos, Dm * d, "act_pos"));
    JPI_TRY(put_block(h, dev, &h->ab, w->ab, true, "ab"));
    JPI_TRY(put_mat(h, dev, &h->fuse_w, w->fuse_w, d * 2 * d, "fuse_w"));
    JPI_TRY(put_vec(h, dev, &h->fuse_b, w->fuse_b, d, "fuse_b"));
    h->jb.resize((size_t)h->J);
    for (int i = 0; i < h->J; ++i) {
        char nm[16];
        snprintf(nm, sizeof(nm), "jb%d", i);
        JPI_TRY(put_block(h, dev, &h->jb[(size_t)i], w->jb[i], true, nm));
    }
    JPI_TRY(put_vec(h, dev, &h->head_ln_w, w->head_ln_w, d, "head_ln_w"));
    JPI_TRY(put_vec(h, dev, &h->head_ln_b, w->head_ln_b, d, "head_ln_b"));
    JPI_TRY(put_mat(h, dev, &h->corr_w, w->corr_w, d * d, "corr_w"));
    JPI_TRY(put_vec(h, dev, &h->corr_b, w->corr_b, d, "corr_b"));
    JPI_TRY(put_vec(h, dev, &h->conf_w, w->conf_w, d, "conf_w"));
    JPI_TRY(put_vec(h, dev, &h->conf_b, w->conf_b, 1, "conf_b"));

    // Weight-only values and activations.
    JPI_TRY(corr_alloc(h, &h->x1b, B * T * d));
    JPI_TRY(corr_alloc(h, &h->qk, M * dv));
    JPI_TRY(corr_alloc(h, &h->t1, B * Dm * d));
    JPI_TRY(corr_alloc(h, &h->xa, B * Dm * d));
    JPI_TRY(corr_alloc(h, &h->ua, B * Dm * d));
    JPI_TRY(corr_alloc(h, &h->kva, B * Dm * 2 * d));
    JPI_TRY(corr_alloc(h, &h->ql, B * d));
    JPI_TRY(corr_alloc(h, &h->ol, B * d));
    JPI_TRY(corr_alloc(h, &h->xl, B * d));
    JPI_TRY(corr_alloc(h, &h->ul, B * d));
    JPI_TRY(corr_alloc(h, &h->hidl, B * F));
    JPI_TRY(corr_alloc(h, &h->xj, B * T * 2 * d));
    JPI_TRY(corr_alloc(h, &h->xf, B * T * d));
    JPI_TRY(corr_alloc(h, &h->u, B * T * d));
    JPI_TRY(corr_alloc(h, &h->qkv, B * T * 3 * d));
    JPI_TRY(corr_alloc(h, &h->o, B * T * d));
    JPI_TRY(corr_alloc(h, &h->hid, B * T * F));
    JPI_TRY(corr_alloc(h, &h->sc, B * M * (size_t)h->Tm));
    JPI_TRY(corr_alloc(h, &h->gs, B * M * dv));
    JPI_TRY(corr_alloc(h, &h->scp, B * (size_t)((dv + CORR_KCHUNK - 1) / CORR_KCHUNK) * M * h->Tm));
    JPI_TRY(corr_alloc(h, &h->gsp, B * (size_t)((h->Tm + CORR_TCHUNK - 1) / CORR_TCHUNK) * M * dv));
    JPI_TRY(corr_alloc(h, reinterpret_cast<float**>(&h->in_vlm), B * (size_t)h->Tm * dv));
    JPI_TRY(corr_alloc(h, &h->in_state, B * (size_t)h->Ti * h->d));
    JPI_TRY(corr_alloc(h, &h->in_act, B * (size_t)h->Dm * h->A));
    JPI_TRY(corr_alloc(h, &h->out_st, B * (size_t)h->Ti * h->d));
    JPI_TRY(corr_alloc(h, &h->out_conf, (size_t)B));
    JPI_CUDA_TRY(cudaStreamCreateWithFlags(&h->cap, cudaStreamNonBlocking));
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_corr_scores<float, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)CORR_SCORES_SMEM));
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_corr_scores<float, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)CORR_SCORES_SMEM));
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_corr_scores<__nv_bfloat16, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)CORR_SCORES_SMEM));
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_corr_scores<__nv_bfloat16, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)CORR_SCORES_SMEM));
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_corr_linear_pipe<4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      4 * LP_ROWS * 2048 * 2));
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_corr_linear_pipe<3>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      3 * LP_ROWS * LP_MAX_IN * 2));
    {
        int dev = 0;
        JPI_CUDA_TRY(cudaGetDevice(&dev));
        JPI_CUDA_TRY(cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, dev));
    }
    JPI_TRY(corr_alloc(h, &h->conf_scratch, B));

    JPI_TRY(prepare(h, nullptr));
    JPI_CUDA_TRY(cudaStreamSynchronize(nullptr));
    return JPI_OK;
}

}  // namespace

namespace {

// The compressor's kernel sequence on `st`: hvlm [batch][n_tokens][dv] -> out [batch][T'][d].
jpi_status enqueue_compress(jpi_corr_handle* h, const void* hvlm, int vlm_is_fp32, int batch, int n_tokens,
                            float* out, cudaStream_t st) {
    const int d = h->d, T = h->Ti, M = h->M, dv = h->dv, rows = batch * T;
    const int nkc = (dv + CORR_KCHUNK - 1) / CORR_KCHUNK, ntc = (n_tokens + CORR_TCHUNK - 1) / CORR_TCHUNK;
    const dim3 gs((unsigned)((n_tokens + 31) / 32), (unsigned)nkc, (unsigned)batch);
    const dim3 gw((unsigned)((dv + 255) / 256), (unsigned)ntc, (unsigned)batch);
    const int red_grid = grid_for((long long)batch * M * dv);
    if (vlm_is_fp32) {
        const float* hv = static_cast<const float*>(hvlm);
        if (dv % 4 == 0 && ((uintptr_t)hv & 15) == 0)
            pdl(st, dim3(gs), dim3(256), CORR_SCORES_SMEM, k_corr_scores<float, true>, h->qk, hv, h->scp, M, n_tokens, dv);
        else
            pdl(st, dim3(gs), dim3(256), CORR_SCORES_SMEM, k_corr_scores<float, false>, h->qk, hv, h->scp, M, n_tokens, dv);
        pdl(st, dim3(batch * M), dim3(256), 0, k_corr_softmax_sum, h->scp, h->sc, M, n_tokens, nkc);
        const bool pair = dv % 2 == 0 && ((uintptr_t)hv & 7) == 0;
        if (M <= 32) {
            if (pair) pdl(st, dim3(gw), dim3(256), 0, k_corr_wsum<float, 16, true>, h->sc, hv, h->gsp, M, n_tokens, dv);
            else pdl(st, dim3(gw), dim3(256), 0, k_corr_wsum<float, 16, false>, h->sc, hv, h->gsp, M, n_tokens, dv);
        } else {
            if (pair) pdl(st, dim3(gw), dim3(256), 0, k_corr_wsum<float, 32, true>, h->sc, hv, h->gsp, M, n_tokens, dv);
            else pdl(st, dim3(gw), dim3(256), 0, k_corr_wsum<float, 32, false>, h->sc, hv, h->gsp, M, n_tokens, dv);
        }
    } else {
        const __nv_bfloat16* hv = static_cast<const __nv_bfloat16*>(hvlm);
        if (dv % 4 == 0 && ((uintptr_t)hv & 7) == 0)
            pdl(st, dim3(gs), dim3(256), CORR_SCORES_SMEM, k_corr_scores<__nv_bfloat16, true>, h->qk, hv, h->scp, M, n_tokens, dv);
        else
            pdl(st, dim3(gs), dim3(256), CORR_SCORES_SMEM, k_corr_scores<__nv_bfloat16, false>, h->qk, hv, h->scp, M, n_tokens, dv);
        pdl(st, dim3(batch * M), dim3(256), 0, k_corr_softmax_sum, h->scp, h->sc, M, n_tokens, nkc);
        const bool pair = dv % 2 == 0 && ((uintptr_t)hv & 3) == 0;
        if (M <= 32) {
            if (pair) pdl(st, dim3(gw), dim3(256), 0, k_corr_wsum<__nv_bfloat16, 16, true>, h->sc, hv, h->gsp, M, n_tokens, dv);
            else pdl(st, dim3(gw), dim3(256), 0, k_corr_wsum<__nv_bfloat16, 16, false>, h->sc, hv, h->gsp, M, n_tokens, dv);
        } else {
            if (pair) pdl(st, dim3(gw), dim3(256), 0, k_corr_wsum<__nv_bfloat16, 32, true>, h->sc, hv, h->gsp, M, n_tokens, dv);
            else pdl(st, dim3(gw), dim3(256), 0, k_corr_wsum<__nv_bfloat16, 32, false>, h->sc, hv, h->gsp, M, n_tokens, dv);
        }
    }
    pdl(st, dim3(red_grid), dim3(256), 0, k_corr_wsum_reduce, h->gsp, h->gs, batch, M, dv, ntc);
    JPI_CUDA_TRY(cudaGetLastError());
    // out_hi = W_v,h g_hi + b_v (head-select rows of gs), then the output projection onto the
    // queries' residual, the MLP, and the output LayerNorm.
    JPI_TRY(linear(h, st, h->gs, dv, h->qf_ca_wv, h->qf_ca_bv, nullptr, 0, h->o, d, rows, dv, d, false, T));
    JPI_TRY(linear(h, st, h->o, d, h->qf_ca_wo, h->qf_ca_bo, h->x1b, d, h->xf, d, rows, d, d, false));
    JPI_TRY(layernorm(h, st, h->xf, d, h->qf_ln3_w, h->qf_ln3_b, h->u, d, rows));
    JPI_TRY(linear(h, st, h->u, d, h->qf_w1, h->qf_b1, nullptr, 0, h->hid, h->F, rows, d, h->F, true));
    JPI_TRY(linear(h, st, h->hid, h->F, h->qf_w2, h->qf_b2, h->xf, d, h->xf, d, rows, h->F, d, false));
    JPI_TRY(layernorm(h, st, h->xf, d, h->qf_lnf_w, h->qf_lnf_b, out, d, rows));
    return JPI_OK;
}

// f_corr's kernel sequence on `st`: state, actions -> out [batch][T'][d], conf [batch].
jpi_status enqueue_predict(jpi_corr_handle* h, const float* state, const float* actions, int batch, int delta,
                           float* out, float* conf, cudaStream_t st) {
    const int d = h->d, T = h->Ti, F = h->F, ra = batch * delta, rows = batch * T;
    const BlockDev& ab = h->ab;
    // Action tokens: MLP, plus the position row of each action.
    JPI_TRY(linear(h, st, actions, h->A, h->act_w1, h->act_b1, nullptr, 0, h->t1, d, ra, h->A, d, true));
    JPI_TRY(linear(h, st, h->t1, d, h->act_w2, h->act_b2, nullptr, 0, h->xa, d, ra, d, d, false));
    pdl(st, dim3(grid_for((long long)ra * d)), dim3(256), 0, k_corr_add_pos, h->xa, h->act_pos, batch, delta, d);
    JPI_CUDA_TRY(cudaGetLastError());
    // Block ab, kept at the last action of each request only: keys and values of every action,
    // the query, attention output, residual and MLP of the last.
    JPI_TRY(layernorm(h, st, h->xa, d, ab.ln1_w, ab.ln1_b, h->ua, d, ra));
    JPI_TRY(linear(h, st, h->ua, d, tw_rows(h, ab.wqkv, (size_t)d, (size_t)d), ab.bqkv + d, nullptr, 0, h->kva,
                   2 * d, ra, d, 2 * d, false));
    const size_t last = (size_t)(delta - 1) * d;
    JPI_TRY(linear(h, st, h->ua + last, delta * d, ab.wqkv, ab.bqkv, nullptr, 0, h->ql, d, batch, d, d, false));
    JPI_TRY(attention(h, st, h->ql, d, h->kva, 2 * d, h->kva + d, 2 * d, h->ol, d, batch, 1, delta));
    JPI_TRY(linear(h, st, h->ol, d, ab.wo, ab.bo, h->xa + last, delta * d, h->xl, d, batch, d, d, false));
    JPI_TRY(layernorm(h, st, h->xl, d, ab.ln2_w, ab.ln2_b, h->ul, d, batch));
    JPI_TRY(linear(h, st, h->ul, d, ab.w1, ab.b1, nullptr, 0, h->hidl, F, batch, d, F, true));
    JPI_TRY(linear(h, st, h->hidl, F, ab.w2, ab.b2, h->xl, d, h->xl, d, batch, F, d, false));
    // Join: [compressed token ; action summary] projected back to the module width.
    pdl(st, dim3(grid_for((long long)rows * 2 * d)), dim3(256), 0, k_corr_join, state, h->xl, h->xj, batch, T, d);
    JPI_CUDA_TRY(cudaGetLastError());
    JPI_TRY(linear(h, st, h->xj, 2 * d, h->fuse_w, h->fuse_b, nullptr, 0, h->xf, d, rows, 2 * d, d, false));
    for (int i = 0; i < h->J; ++i) JPI_TRY(block(h, st, h->jb[(size_t)i], h->xf, batch, T));
    // Heads.
    JPI_TRY(layernorm(h, st, h->xf, d, h->head_ln_w, h->head_ln_b, h->u, d, rows));
    JPI_TRY(linear(h, st, h->u, d, h->corr_w, h->corr_b, nullptr, 0, out, d, rows, d, d, false));
    pdl(st, dim3(batch), dim3(256), 0, k_corr_confidence, h->u, h->conf_w, h->conf_b, conf, T, d);
    JPI_CUDA_TRY(cudaGetLastError());
    return JPI_OK;
}

// The graph of one call shape, captured on the handle's own stream the first time it is asked for.
template <typename F>
jpi_status corr_graph(jpi_corr_handle* h, std::tuple<int, int, int, int> key, F&& enqueue, cudaGraphExec_t* out) {
    auto it = h->graphs.find(key);
    if (it != h->graphs.end()) {
        *out = it->second;
        return JPI_OK;
    }
    cudaGraph_t g = nullptr;
    JPI_CUDA_TRY(cudaStreamBeginCapture(h->cap, cudaStreamCaptureModeThreadLocal));
    const jpi_status s = enqueue(h->cap);
    const cudaError_t e = cudaStreamEndCapture(h->cap, &g);
    if (s != JPI_OK) {
        if (g) cudaGraphDestroy(g);
        return s;
    }
    if (e != cudaSuccess) return cfail(JPI_ERR_CUDA, "graph capture failed: %s", cudaGetErrorString(e));
    cudaGraphExec_t ex = nullptr;
    const cudaError_t ei = cudaGraphInstantiate(&ex, g, 0);
    cudaGraphDestroy(g);
    if (ei != cudaSuccess) return cfail(JPI_ERR_CUDA, "graph instantiate failed: %s", cudaGetErrorString(ei));
    h->graphs[key] = ex;
    *out = ex;
    return JPI_OK;
}

}  // namespace

extern "C" {

JPI_API jpi_status jpi_corr_create(const jpi_corr_config* cfg, const jpi_corr_weights* w,
                                   jpi_corr_handle** out) {
    jpi::clear_error();
    if (!out) return cfail(JPI_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    if (!cfg || !w) return cfail(JPI_ERR_INVALID_ARG, "config or weights is NULL");
    JPI_TRY(check_corr_config(cfg));
    if (cfg->n_joint > 0 && !w->jb) return cfail(JPI_ERR_INVALID_ARG, "joint blocks (jb) are NULL");
    jpi_corr_handle* h = new (std::nothrow) jpi_corr_handle();
    if (!h) return cfail(JPI_ERR_OOM, "host allocation failed");
    const jpi_status s = setup(h, cfg, w);
    if (s != JPI_OK) {
        cudaStreamSynchronize(nullptr);   // let any conversion in flight finish before its buffers go
        cudaGetLastError();
        if (h->cap) cudaStreamDestroy(h->cap);
        for (void* p : h->allocs) cudaFree(p);
        delete h;
        return s;
    }
    *out = h;
    return JPI_OK;
}

JPI_API jpi_status jpi_corr_destroy(jpi_corr_handle* h) {
    jpi::clear_error();
    if (!h) return JPI_OK;
    cudaDeviceSynchronize();
    for (auto& kv : h->graphs) cudaGraphExecDestroy(kv.second);
    if (h->cap) cudaStreamDestroy(h->cap);
    for (void* p : h->allocs) cudaFree(p);
    cudaGetLastError();
    delete h;
    return JPI_OK;
}

JPI_API jpi_status jpi_corr_compress(jpi_corr_handle* h, const void* h_vlm, int vlm_is_fp32, int batch,
                                     int n_tokens, float* out_state, void* stream) {
    jpi::clear_error();
    if (!h) return cfail(JPI_ERR_INVALID_ARG, "handle is NULL");
    if (!h_vlm || !out_state) return cfail(JPI_ERR_INVALID_ARG, "NULL input or output");
    if (batch < 1 || n_tokens < 1) return cfail(JPI_ERR_INVALID_ARG, "batch and n_tokens must be >= 1");
    if (batch > h->B || n_tokens > h->Tm)
        return cfail(JPI_ERR_SHAPE, "batch %d / n_tokens %d exceed the maxima %d / %d", batch, n_tokens, h->B,
                     h->Tm);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const size_t in_bytes = (size_t)batch * n_tokens * h->dv * (vlm_is_fp32 ? 4 : 2);
    cudaGraphExec_t ex = nullptr;
    JPI_TRY(corr_graph(h, std::make_tuple(0, batch, n_tokens, vlm_is_fp32 ? 1 : 0),
                       [&](cudaStream_t cs) {
                           return enqueue_compress(h, h->in_vlm, vlm_is_fp32, batch, n_tokens, h->out_st, cs);
                       },
                       &ex));
    JPI_CUDA_TRY(cudaMemcpyAsync(h->in_vlm, h_vlm, in_bytes, cudaMemcpyDeviceToDevice, st));
    JPI_CUDA_TRY(cudaGraphLaunch(ex, st));
    JPI_CUDA_TRY(cudaMemcpyAsync(out_state, h->out_st, (size_t)batch * h->Ti * h->d * sizeof(float),
                                 cudaMemcpyDeviceToDevice, st));
    return JPI_OK;
}

JPI_API jpi_status jpi_corr_predict(jpi_corr_handle* h, const float* state, const float* actions, int batch,
                                    int delta, float* out_state, float* out_confidence, void* stream) {
    jpi::clear_error();
    if (!h) return cfail(JPI_ERR_INVALID_ARG, "handle is NULL");
    if (!state || !actions || !out_state) return cfail(JPI_ERR_INVALID_ARG, "NULL input or output");
    if (batch < 1 || delta < 1) return cfail(JPI_ERR_INVALID_ARG, "batch and delta must be >= 1");
    if (batch > h->B || delta > h->Dm)
        return cfail(JPI_ERR_SHAPE, "batch %d / delta %d exceed the maxima %d / %d", batch, delta, h->B, h->Dm);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaGraphExec_t ex = nullptr;
    JPI_TRY(corr_graph(h, std::make_tuple(1, batch, delta, 0),
                       [&](cudaStream_t cs) {
                           return enqueue_predict(h, h->in_state, h->in_act, batch, delta, h->out_st, h->out_conf, cs);
                       },
                       &ex));
    const size_t state_bytes = (size_t)batch * h->Ti * h->d * sizeof(float);
    JPI_CUDA_TRY(cudaMemcpyAsync(h->in_state, state, state_bytes, cudaMemcpyDeviceToDevice, st));
    JPI_CUDA_TRY(cudaMemcpyAsync(h->in_act, actions, (size_t)batch * delta * h->A * sizeof(float),
                                 cudaMemcpyDeviceToDevice, st));
    JPI_CUDA_TRY(cudaGraphLaunch(ex, st));
    JPI_CUDA_TRY(cudaMemcpyAsync(out_state, h->out_st, state_bytes, cudaMemcpyDeviceToDevice, st));
    if (out_confidence)
        JPI_CUDA_TRY(cudaMemcpyAsync(out_confidence, h->out_conf, (size_t)batch * sizeof(float),
                                     cudaMemcpyDeviceToDevice, st));
    return JPI_OK;
}

JPI_API jpi_status jpi_corr_memory_usage(const jpi_corr_handle* h, long long* bytes) {
    jpi::clear_error();
    if (!h || !bytes) return cfail(JPI_ERR_INVALID_ARG, "handle or bytes is NULL");
    *bytes = (long long)h->bytes;
    return JPI_OK;
}

}  // extern "C"
