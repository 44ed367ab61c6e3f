// CUDA-core kernels: time conditioning, token embedding, the fp32 verification path of every
// layer op, the final norm + action-out projection + Euler update, and KV-store conversion.
//
// Every reduction here runs in a fixed order (fixed per-thread strides, then a fixed shuffle
// tree), so results are bitwise reproducible run to run.

#include "jpi_internal.h"
#include "tc_path.h"
#include "ptx.h"

#include <cmath>
#include <type_traits>

namespace jpi {
namespace {

template <typename T> __device__ __forceinline__ float ldf(const T* p);
template <> __device__ __forceinline__ float ldf<float>(const float* p) { return *p; }
template <> __device__ __forceinline__ float ldf<__nv_bfloat16>(const __nv_bfloat16* p) {
    return __bfloat162float(*p);
}
template <typename T> __device__ __forceinline__ T cvt(float v);
template <> __device__ __forceinline__ float cvt<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 cvt<__nv_bfloat16>(float v) {
    return __float2bfloat16_rn(v);
}

__device__ __forceinline__ float swishf(float z) { return z / (1.f + expf(-z)); }

// GELU, tanh form (Gemma's MLP activation).
__device__ __forceinline__ float gelu_tanhf(float y) {
    const float k0 = 0.7978845608028654f;   // sqrt(2 / pi)
    return 0.5f * y * (1.f + tanhf(k0 * (y + 0.044715f * y * y * y)));
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Sum over a block of up to 1024 threads (blockDim a multiple of 32), fixed order.
__device__ float block_sum(float v, float* scratch /* >= 32 floats */) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    v = warp_sum(v);
    __syncthreads();
    if (lane == 0) scratch[warp] = v;
    __syncthreads();
    float t = lane < nw ? scratch[lane] : 0.f;
    t = warp_sum(t);
    return t;
}

// ---------------------------------------------------------------------------------------------
// Time conditioning: flow time enters the expert only through a sinusoidal embedding followed
// by a two-layer swish MLP; the per-layer modulation vectors are a linear map of the result.
// All of it depends on t alone, so it is evaluated once per call for every step time.

// Grid (steps, ceil(half / blockDim)): one frequency i of one step time per thread (the fp64
// pow/sin/cos are slow on this GPU; spread over the grid they run side by side).
__global__ void k_time_embed(float* temb, int nsteps, int dt, double pmin, double pmax,
                             double t_override) {
    const int k = blockIdx.x;
    const double t = t_override >= 0.0 ? t_override : (double)k / (double)nsteps;
    const int half = dt / 2;
    for (int i = blockIdx.y * blockDim.x + threadIdx.x; i < half; i += gridDim.y * blockDim.x) {
        const double frac = (double)i / (double)(half - 1);
        const double period = pmin * pow(pmax / pmin, frac);
        const double theta = 2.0 * 3.14159265358979323846 * t / period;
        temb[(size_t)k * dt + i] = (float)sin(theta);
        temb[(size_t)k * dt + half + i] = (float)cos(theta);
    }
}

// Y[n][r] = act(sum_k W[r][k] X[n][k] + b[r]) for n < N (<= 8 per pass), r < R.
// One warp per output row; X lives in shared memory.
template <typename TW, bool SWISH>
__global__ void k_gemv_multi(const TW* __restrict__ Wm, const float* __restrict__ bias,
                             const float* __restrict__ X, float* __restrict__ Y, int R, int K,
                             int N) {
    extern __shared__ float xs[];
    // Eight loads of each thread in flight before their stores (one at a time, every store would
    // hold the next load back for a full round trip).
    for (int i0 = threadIdx.x; i0 < N * K; i0 += 8 * blockDim.x) {
        float v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int i = i0 + u * blockDim.x;
            v[u] = i < N * K ? X[i] : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int i = i0 + u * blockDim.x;
            if (i < N * K) xs[i] = v[u];
        }
    }
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int nwarps = (gridDim.x * blockDim.x) >> 5;
    for (int r = warp; r < R; r += nwarps) {
        const TW* wr = Wm + (size_t)r * K;
        for (int n0 = 0; n0 < N; n0 += 8) {
            float acc[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) acc[j] = 0.f;
            // Eight weights of the row loaded together, then their products in k order.
            for (int k0 = lane; k0 < K; k0 += 32 * 8) {
                float wv[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int k = k0 + 32 * u;
                    wv[u] = k < K ? ldf(wr + k) : 0.f;
                }
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int k = k0 + 32 * u;
                    if (k < K) {
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            if (n0 + j < N) acc[j] = fmaf(wv[u], xs[(n0 + j) * K + k], acc[j]);
                    }
                }
            }
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const float s = warp_sum(acc[j]);
                if (lane == 0 && n0 + j < N) {
                    const float y = s + bias[r];
                    Y[(size_t)(n0 + j) * R + r] = SWISH ? swishf(y) : y;
                }
            }
        }
    }
}

// Y[n][r] = sum_k W[r][k] X[n][k] + b[r] for all n < NG step times at once: the stacked
// modulation matrix (6 L + 2) W rows is streamed from HBM exactly once per call. Each thread
// owns MOD_RT consecutive rows; per 16-wide K slab it loads 32 bytes of every row (full
// sectors) and reads each X value as a shared-memory broadcast, so the inner loop is FMAs.
constexpr int MOD_RT = 4;

template <typename TW> struct Slab;                 // 16 consecutive weights of one row
template <> struct Slab<__nv_bfloat16> {
    uint4 v[2];
    __device__ __forceinline__ void load(const __nv_bfloat16* p) {
        v[0] = __ldg((const uint4*)p);
        v[1] = __ldg((const uint4*)p + 1);
    }
    __device__ __forceinline__ float get(int i) const {
        const uint32_t u = (&v[0].x)[i >> 1];
        return __uint_as_float((i & 1) ? (u & 0xFFFF0000u) : (u << 16));
    }
};
template <> struct Slab<float> {
    float4 v[4];
    __device__ __forceinline__ void load(const float* p) {
#pragma unroll
        for (int i = 0; i < 4; ++i) v[i] = __ldg((const float4*)p + i);
    }
    __device__ __forceinline__ float get(int i) const { return (&v[0].x)[i]; }
};

template <typename TW, int NG>
__global__ void __launch_bounds__(256) k_mod_gemv(const TW* __restrict__ Wm, const float* __restrict__ bias,
                                                   const float* __restrict__ X, float* __restrict__ Y,
                                                   int R, int K) {
    extern __shared__ float xs[];                     // [NG][K]
    for (int i = threadIdx.x; i < NG * K; i += blockDim.x) xs[i] = X[i];
    __syncthreads();
    const int r0 = (blockIdx.x * blockDim.x + threadIdx.x) * MOD_RT;
    if (r0 >= R) return;
    float acc[MOD_RT][NG];
#pragma unroll
    for (int rr = 0; rr < MOD_RT; ++rr)
#pragma unroll
        for (int n = 0; n < NG; ++n) acc[rr][n] = 0.f;
    const TW* rowp[MOD_RT];
#pragma unroll
    for (int rr = 0; rr < MOD_RT; ++rr) rowp[rr] = Wm + (size_t)min(r0 + rr, R - 1) * K;
    Slab<TW> cur[MOD_RT], nxt[MOD_RT];
#pragma unroll
    for (int rr = 0; rr < MOD_RT; ++rr) cur[rr].load(rowp[rr]);
    for (int k0 = 0; k0 < K; k0 += 16) {
        if (k0 + 16 < K) {
#pragma unroll
            for (int rr = 0; rr < MOD_RT; ++rr) nxt[rr].load(rowp[rr] + k0 + 16);
        }
#pragma unroll
        for (int kk = 0; kk < 16; ++kk) {
            float w[MOD_RT];
#pragma unroll
            for (int rr = 0; rr < MOD_RT; ++rr) w[rr] = cur[rr].get(kk);
#pragma unroll
            for (int n = 0; n < NG; ++n) {
                const float xv = xs[n * K + k0 + kk];
#pragma unroll
                for (int rr = 0; rr < MOD_RT; ++rr) acc[rr][n] = fmaf(w[rr], xv, acc[rr][n]);
            }
        }
#pragma unroll
        for (int rr = 0; rr < MOD_RT; ++rr) cur[rr] = nxt[rr];
    }
#pragma unroll
    for (int n = 0; n < NG; ++n)
#pragma unroll
        for (int rr = 0; rr < MOD_RT; ++rr)
            if (r0 + rr < R) Y[(size_t)n * R + r0 + rr] = acc[rr][n] + bias[r0 + rr];
}

// ---------------------------------------------------------------------------------------------
// Token embedding: row 0 of each request is the state token, rows 1..nctx-1 the correction
// items (context tokens, taken as given), then the C action tokens.
// Block = 128 features of one token. For the tensor-core path it also writes the operand of
// the first layer's norm-fed projection (xs = bf16((1 + sigma) * h) at row xs_row(m), and beta in
// the last row of tile m while m < xs_tiles) and that slice's sum of squares (ss[slice][m]).
__global__ void __launch_bounds__(128) k_embed(
    float* __restrict__ hres, __nv_bfloat16* __restrict__ xs, const float* __restrict__ sigma,
    const float* __restrict__ beta, float* __restrict__ ss, int ss_ld,
    const float* __restrict__ state,
    const float* __restrict__ x, const float* __restrict__ Ws, const float* __restrict__ bs,
    const float* __restrict__ Wa, const float* __restrict__ ba, const float* __restrict__ corr, int nctx,
    int S, int C, int W, int Sd, int A) {
    __shared__ float scratch[32];
    const int m = blockIdx.y;
    const int b = m / S, i = m % S;
    const float* in = nullptr;
    const float* Wm = nullptr;
    const float* bias = nullptr;
    int K = 0;
    if (i == 0) {
        in = state + (size_t)b * Sd; Wm = Ws; bias = bs; K = Sd;
    } else if (i >= nctx) {
        in = x + ((size_t)b * C + (i - nctx)) * A; Wm = Wa; bias = ba; K = A;
    }
    const int n = blockIdx.x * 128 + threadIdx.x;
    // Everything but x (the previous step's actions) is ready before the dependency wait: the
    // first EMB_K weights of this feature's row, its bias and the norm's scale and shift.
    constexpr int EMB_K = 32;
    float wv[EMB_K];
    float bv = 0.f, sg = 0.f, bt = 0.f;
    const bool lin = n < W && !(i > 0 && i < nctx);
    if (lin) {
#pragma unroll
        for (int k = 0; k < EMB_K; ++k) wv[k] = k < K ? Wm[(size_t)n * K + k] : 0.f;
        bv = bias[n];
    }
    if (n < W && xs) {
        sg = sigma[n];
        bt = beta[n];
    }
    // Launched with programmatic dependent launch: x comes from the previous step's final kernel;
    // the next kernel may start its weight prefetch at once.
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    float v = 0.f;
    if (n < W) {
        if (!lin) {
            v = corr[((size_t)b * (nctx - 1) + (i - 1)) * W + n];
        } else {
            // The inputs of this row loaded together, then summed in k order.
            float acc = 0.f;
            float iv[EMB_K];
#pragma unroll
            for (int k = 0; k < EMB_K; ++k) iv[k] = k < K ? in[k] : 0.f;
#pragma unroll
            for (int k = 0; k < EMB_K; ++k)
                if (k < K) acc = fmaf(wv[k], iv[k], acc);
            for (int k = EMB_K; k < K; ++k) acc = fmaf(Wm[(size_t)n * K + k], in[k], acc);
            v = acc + bv;
        }
        hres[(size_t)m * W + n] = v;
        if (xs) {
            xs[(size_t)xs_row(m) * W + n] = __float2bfloat16_rn((1.f + sg) * v);
            if (m < xs_tiles(gridDim.y)) xs[((size_t)m * 64 + 63) * W + n] = __float2bfloat16_rn(bt);
        }
    }
    if (ss) {
        const float t = block_sum(v * v, scratch);
        if (threadIdx.x == 0) ss[(size_t)blockIdx.x * ss_ld + m] = t;
    }
}

// ---------------------------------------------------------------------------------------------
// Adaptive RMSNorm of one token row: u = h / sqrt(mean(h^2) + eps) * (1 + sigma) + beta.
template <typename TA>
__global__ void k_rms_mod(const float* __restrict__ hres, const float* __restrict__ sigma,
                          const float* __restrict__ beta, TA* __restrict__ out, int W, int ldo,
                          float eps) {
    __shared__ float scratch[32];
    const int m = blockIdx.x;
    const float* hr = hres + (size_t)m * W;
    float ss = 0.f;
    for (int k = threadIdx.x; k < W; k += blockDim.x) ss = fmaf(hr[k], hr[k], ss);
    ss = block_sum(ss, scratch);
    const float rinv = rsqrtf(ss / (float)W + eps);
    for (int k = threadIdx.x; k < W; k += blockDim.x)
        out[(size_t)m * ldo + k] = cvt<TA>(hr[k] * rinv * (1.f + sigma[k]) + beta[k]);
}

// ---------------------------------------------------------------------------------------------
// CUDA-core GEMM Y[m][n] = sum_k X[m][k] W[n][k] with three epilogues:
//   STORE  Y[m][n] = y
//   RESID  Y[m][n] += gamma[n] * y            (gated residual update of h)
//   GEGLU  Z[m][n] = gelu_tanh(y_gate) * y_up (second weight matrix W2 = up)
enum { EPI_STORE = 0, EPI_RESID = 1, EPI_GEGLU = 2 };

constexpr int GB_M = 64, GB_N = 64, GB_K = 16;

template <typename TA, typename TW, int EPI>
__global__ void __launch_bounds__(256) k_gemm_simt(
    const TA* __restrict__ X, int ldx, const TW* __restrict__ W1, const TW* __restrict__ W2,
    int M, int N, int K, float* __restrict__ Y, int ldy, const float* __restrict__ gamma,
    TA* __restrict__ Z, int ldz) {
    __shared__ float xs[GB_K][GB_M + 4];
    __shared__ float ws[GB_K][GB_N + 4];
    __shared__ float us[(EPI == EPI_GEGLU) ? GB_K : 1][GB_N + 4];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int m0 = blockIdx.y * GB_M, n0 = blockIdx.x * GB_N;
    float acc[4][4] = {}, acc2[4][4] = {};
    for (int k0 = 0; k0 < K; k0 += GB_K) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int idx = tid + e * 256;          // 0..1023 over a 64 x 16 tile
            const int r = idx >> 4, kk = idx & 15;
            const int gm = m0 + r, gn = n0 + r, gk = k0 + kk;
            xs[kk][r] = (gm < M && gk < K) ? ldf(X + (size_t)gm * ldx + gk) : 0.f;
            ws[kk][r] = (gn < N && gk < K) ? ldf(W1 + (size_t)gn * K + gk) : 0.f;
            if (EPI == EPI_GEGLU)
                us[kk][r] = (gn < N && gk < K) ? ldf(W2 + (size_t)gn * K + gk) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < GB_K; ++kk) {
            float a[4], bw[4], bu[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = xs[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) bw[j] = ws[kk][tx * 4 + j];
            if (EPI == EPI_GEGLU) {
#pragma unroll
                for (int j = 0; j < 4; ++j) bu[j] = us[kk][tx * 4 + j];
            }
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    acc[i][j] = fmaf(a[i], bw[j], acc[i][j]);
                    if (EPI == EPI_GEGLU) acc2[i][j] = fmaf(a[i], bu[j], acc2[i][j]);
                }
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int m = m0 + ty * 4 + i;
        if (m >= M) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int n = n0 + tx * 4 + j;
            if (n >= N) continue;
            if (EPI == EPI_STORE) {
                Y[(size_t)m * ldy + n] = acc[i][j];
            } else if (EPI == EPI_RESID) {
                Y[(size_t)m * ldy + n] += gamma[n] * acc[i][j];
            } else {
                Z[(size_t)m * ldz + n] = cvt<TA>(gelu_tanhf(acc[i][j]) * acc2[i][j]);
            }
        }
    }
}

// ---------------------------------------------------------------------------------------------
// Rotary encoding of the suffix q and k at positions P + i (rotate-half pairs (d, d + D/2)),
// then q to the query buffer and k, v into the KV store's suffix tail of this layer.
template <typename TQ, typename TKV>
__global__ void k_qkv_post(const float* __restrict__ qkv, TQ* __restrict__ q,
                           TKV* __restrict__ kst, TKV* __restrict__ vst,
                           const float2* __restrict__ rope, int S, int H, int D, int P,
                           int kv_rows) {
    const int m = blockIdx.x;
    const int b = m / S, i = m % S, pos = P + i;
    const int hd = D / 2, QKVd = (H + 2) * D;
    const float* row = qkv + (size_t)m * QKVd;
    for (int idx = threadIdx.x; idx < (H + 1) * hd; idx += blockDim.x) {
        const int hh = idx / hd, d = idx % hd;       // hh == H is the key head
        const float x1 = row[hh * D + d], x2 = row[hh * D + d + hd];
        float c = 1.f, s = 0.f;
        if (rope) { const float2 cs = rope[(size_t)pos * hd + d]; c = cs.x; s = cs.y; }
        const float y1 = x1 * c - x2 * s, y2 = x2 * c + x1 * s;
        if (hh < H) {
            q[(size_t)m * H * D + hh * D + d] = cvt<TQ>(y1);
            q[(size_t)m * H * D + hh * D + d + hd] = cvt<TQ>(y2);
        } else {
            kst[((size_t)b * kv_rows + pos) * D + d] = cvt<TKV>(y1);
            kst[((size_t)b * kv_rows + pos) * D + d + hd] = cvt<TKV>(y2);
        }
    }
    for (int d = threadIdx.x; d < D; d += blockDim.x)
        vst[((size_t)b * kv_rows + pos) * D + d] = cvt<TKV>(row[(H + 1) * D + d]);
}

// ---------------------------------------------------------------------------------------------
// Attention of one suffix token (all H heads, one warp each) over [prefix ; suffix] keys of
// the single KV head. The state and context rows (i < nctx) see the prefix and each other;
// action rows see all.
// Online softmax over chunks of 32 keys staged in shared memory.
constexpr int ATT_MAXD = 256;

template <typename TQ, typename TKV, typename TO>
__global__ void k_attn_simt(const TQ* __restrict__ q, const TKV* __restrict__ kst,
                            const TKV* __restrict__ vst, TO* __restrict__ o, int S, int H, int D,
                            int P, int kv_rows, int nctx, float scale) {
    extern __shared__ float sm[];
    float* qs = sm;                      // [H][D]
    float* ks = qs + H * D;              // [32][D + 1]
    float* vs = ks + 32 * (D + 1);       // [32][D]
    const int m = blockIdx.x;
    const int b = m / S, i = m % S;
    const int nvis = (i < nctx) ? P + nctx : P + S;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int idx = threadIdx.x; idx < H * D; idx += blockDim.x)
        qs[idx] = ldf(q + (size_t)m * H * D + idx);
    const int nd = D / 32;
    float acc[ATT_MAXD / 32];
#pragma unroll
    for (int j = 0; j < ATT_MAXD / 32; ++j) acc[j] = 0.f;
    float mx = -INFINITY, l = 0.f;
    const TKV* kb = kst + (size_t)b * kv_rows * D;
    const TKV* vb = vst + (size_t)b * kv_rows * D;
    for (int key0 = 0; key0 < nvis; key0 += 32) {
        __syncthreads();
        for (int idx = threadIdx.x; idx < 32 * D; idx += blockDim.x) {
            const int r = idx / D, d = idx % D;
            const bool ok = key0 + r < nvis;
            ks[r * (D + 1) + d] = ok ? ldf(kb + (size_t)(key0 + r) * D + d) : 0.f;
            vs[r * D + d] = ok ? ldf(vb + (size_t)(key0 + r) * D + d) : 0.f;
        }
        __syncthreads();
        const float* qh = qs + warp * D;
        float s = -INFINITY;
        if (key0 + lane < nvis) {
            float dot = 0.f;
            for (int d = 0; d < D; ++d) dot = fmaf(qh[d], ks[lane * (D + 1) + d], dot);
            s = dot * scale;
        }
        const float cmax = warp_max(s);
        const float nmx = fmaxf(mx, cmax);
        const float corr = (mx == -INFINITY) ? 0.f : expf(mx - nmx);
        const float p = (s == -INFINITY) ? 0.f : expf(s - nmx);
        l = l * corr + warp_sum(p);
#pragma unroll
        for (int j = 0; j < ATT_MAXD / 32; ++j) acc[j] *= corr;
        for (int jj = 0; jj < 32; ++jj) {
            const float pj = __shfl_sync(0xffffffffu, p, jj);
#pragma unroll
            for (int j = 0; j < ATT_MAXD / 32; ++j)
                if (j < nd) acc[j] = fmaf(pj, vs[jj * D + lane + 32 * j], acc[j]);
        }
        mx = nmx;
    }
    const float inv = 1.f / l;
#pragma unroll
    for (int j = 0; j < ATT_MAXD / 32; ++j)
        if (j < nd) o[(size_t)m * H * D + warp * D + lane + 32 * j] = cvt<TO>(acc[j] * inv);
}

// ---------------------------------------------------------------------------------------------
// Final adaptive RMSNorm of an action row, velocity v = u W_out^T + b_out, Euler update
// x <- x + delta v (or, for a single forward, v itself).
// One CTA of FIN_THREADS per action row. The row's values (FIN_CAP per thread at most, all loads
// in flight together) give the norm; the normalised row goes to shared memory; then thread t
// takes output a0 + t / 8 over the 16-byte column chunks t mod 8, t mod 8 + 8, .. (a group of 8
// threads reads 128 contiguous bytes per step) and the group adds its 8 partial sums.
constexpr int FIN_THREADS = 256;
constexpr int FIN_CAP = 16;   // W <= 4096
__global__ void __launch_bounds__(FIN_THREADS) k_final(const float* __restrict__ hres, const float* __restrict__ sigma,
                        const float* __restrict__ beta, const float* __restrict__ Wout,
                        const float* __restrict__ bout, float* __restrict__ x,
                        float* __restrict__ vout, float* __restrict__ outcopy, int S, int nctx, int C,
                        int W, int A, float eps, float delta) {
    extern __shared__ float us[];        // [W]
    __shared__ float scratch[32];
    const int tid = threadIdx.x;
    const int bj = blockIdx.x;           // request b, action j
    const int b = bj / C, j = bj % C;
    // The modulation (scale, shift) of this thread's features, before the dependency wait.
    float sg[FIN_CAP], bt[FIN_CAP];
#pragma unroll
    for (int q = 0; q < FIN_CAP; ++q) {
        const int k = tid + FIN_THREADS * q;
        sg[q] = k < W ? sigma[k] : 0.f;
        bt[q] = k < W ? beta[k] : 0.f;
    }
    // Launched with programmatic dependent launch: h comes from the last layer's down projection.
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    const float* hr = hres + ((size_t)b * S + nctx + j) * W;
    float hv[FIN_CAP];
#pragma unroll
    for (int q = 0; q < FIN_CAP; ++q) {
        const int k = tid + FIN_THREADS * q;
        hv[q] = k < W ? hr[k] : 0.f;
    }
    float ss = 0.f;
#pragma unroll
    for (int q = 0; q < FIN_CAP; ++q) ss = fmaf(hv[q], hv[q], ss);
    for (int k = tid + FIN_THREADS * FIN_CAP; k < W; k += FIN_THREADS) ss = fmaf(hr[k], hr[k], ss);   // W > 4096
    ss = block_sum(ss, scratch);
    const float rinv = rsqrtf(ss / (float)W + eps);
#pragma unroll
    for (int q = 0; q < FIN_CAP; ++q) {
        const int k = tid + FIN_THREADS * q;
        if (k < W) us[k] = hv[q] * rinv * (1.f + sg[q]) + bt[q];
    }
    for (int k = tid + FIN_THREADS * FIN_CAP; k < W; k += FIN_THREADS)
        us[k] = hr[k] * rinv * (1.f + sigma[k]) + beta[k];
    __syncthreads();
    const int ks = tid & 7;
    const int n4 = W >> 2;   // W is a multiple of 32 (checked at create)
    const float4* us4 = reinterpret_cast<const float4*>(us);
    for (int a0 = 0; a0 < A; a0 += FIN_THREADS / 8) {
        const int a = a0 + (tid >> 3);
        float acc = 0.f;
        if (a < A) {
            const float4* wr = reinterpret_cast<const float4*>(Wout + (size_t)a * W);
#pragma unroll 8
            for (int c = ks; c < n4; c += 8) {
                const float4 w4 = __ldg(wr + c), u4 = us4[c];
                acc = fmaf(u4.x, w4.x, fmaf(u4.y, w4.y, fmaf(u4.z, w4.z, fmaf(u4.w, w4.w, acc))));
            }
        }
        acc += __shfl_xor_sync(0xffffffffu, acc, 1);
        acc += __shfl_xor_sync(0xffffffffu, acc, 2);
        acc += __shfl_xor_sync(0xffffffffu, acc, 4);
        if (ks == 0 && a < A) {
            const float v = acc + bout[a];
            const size_t idx = (size_t)bj * A + a;
            if (vout) vout[idx] = v;
            if (x) {
                const float xn = x[idx] + delta * v;
                x[idx] = xn;
                if (outcopy) outcopy[idx] = xn;
            }
        }
    }
}

// ---------------------------------------------------------------------------------------------
// Prefix KV into the store: src [batch][P][D] (fp32 or bf16) -> dst [batch][kv_rows][D].
template <typename TS, typename TD>
__global__ void k_convert_kv(const TS* __restrict__ src, TD* __restrict__ dst, int P, int D,
                             int kv_rows, long long total) {
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x) {
        const long long d = idx % D, p = (idx / D) % P, b = idx / ((long long)D * P);
        dst[((size_t)b * kv_rows + p) * D + d] = cvt<TD>(ldf(src + idx));
    }
}

// Launch with programmatic dependent launch when the handle uses it (the kernel waits for its
// predecessor with griddepcontrol.wait before reading what that wrote); a failed launch leaves its
// error for check_launch.
template <typename... KArgs, typename... Args>
void launch_pdl(const jpi_handle* h, dim3 grid, dim3 block, size_t smem, cudaStream_t st, void (*k)(KArgs...),
                Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at;
    at.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at.val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = &at;
    cfg.numAttrs = h->pdl ? 1 : 0;
    (void)cudaLaunchKernelEx(&cfg, k, args...);
}

inline jpi_status check_launch(const char* what) {
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_error("launch of %s failed: %s", what, cudaGetErrorString(e));
        return JPI_ERR_CUDA;
    }
    return JPI_OK;
}

inline int grid_for(long long n, int block, int cap = 4096) {
    long long g = (n + block - 1) / block;
    return (int)(g < 1 ? 1 : (g > cap ? cap : g));
}

// One sub-step of layer l: 2 norm + QKV + rotary, 3 attention, 4 O-proj + residual,
// 5 norm + gate/up + GeGLU, 6 down-proj + residual.
template <typename T>
jpi_status op_simt(jpi_handle* h, int op, int l, int step, int B, int C, cudaStream_t st) {
    const int S = C + h->n_ctx(), Mt = B * S, W = h->W, F = h->F, HD = h->HD, D = h->D;
    const float* ms = h->mods + (size_t)step * mod_rows(h->L) * W + (size_t)6 * l * W;
    const LayerPlain* lwp = (size_t)l < h->plain.size() ? &h->plain[l] : nullptr;
    T* act = (T*)h->act;
    const size_t kv_layer = (size_t)l * h->maxB * h->kv_rows * D;
    T* kst = (T*)h->kv_k + kv_layer;
    T* vst = (T*)h->kv_v + kv_layer;
    const float eps = h->cfg.rms_eps;
    const dim3 blk(256);
    const int mtiles = (Mt + GB_M - 1) / GB_M;
    if (op != 3 && !lwp) {
        set_error("layer %d has no CUDA-core weights", l);
        return JPI_ERR_INVALID_ARG;
    }
    switch (op) {
        case 2:
            k_rms_mod<T><<<Mt, blk, 0, st>>>(h->h, ms, ms + W, act, W, W, eps);
            k_gemm_simt<T, T, EPI_STORE><<<dim3((h->QKV + GB_N - 1) / GB_N, mtiles), blk, 0, st>>>(
                act, W, (const T*)lwp->wqkv, nullptr, Mt, h->QKV, W, h->qkv, h->QKV, nullptr, nullptr, 0);
            k_qkv_post<T, T><<<Mt, blk, 0, st>>>(h->qkv, (T*)h->q, kst, vst, h->rope_tab, S, h->H, D,
                                                 h->cur_prefix, h->kv_rows);
            break;
        case 3: {
            const size_t att_smem = sizeof(float) * ((size_t)h->H * D + 32 * (D + 1) + 32 * D);
            k_attn_simt<T, T, T><<<Mt, 32 * h->H, att_smem, st>>>(
                (const T*)h->q, kst, vst, (T*)h->o, S, h->H, D, h->cur_prefix, h->kv_rows, h->n_ctx(),
                1.f / sqrtf((float)D));
            break;
        }
        case 4:
            k_gemm_simt<T, T, EPI_RESID><<<dim3((W + GB_N - 1) / GB_N, mtiles), blk, 0, st>>>(
                (const T*)h->o, HD, (const T*)lwp->wo, nullptr, Mt, W, HD, h->h, W, ms + 2 * W, nullptr, 0);
            break;
        case 5:
            k_rms_mod<T><<<Mt, blk, 0, st>>>(h->h, ms + 3 * W, ms + 4 * W, act, W, W, eps);
            k_gemm_simt<T, T, EPI_GEGLU><<<dim3((F + GB_N - 1) / GB_N, mtiles), blk, 0, st>>>(
                act, W, (const T*)lwp->wg, (const T*)lwp->wu, Mt, F, W, nullptr, 0, nullptr, (T*)h->z, F);
            break;
        case 6:
            k_gemm_simt<T, T, EPI_RESID><<<dim3((W + GB_N - 1) / GB_N, mtiles), blk, 0, st>>>(
                (const T*)h->z, F, (const T*)lwp->wd, nullptr, Mt, W, F, h->h, W, ms + 5 * W, nullptr, 0);
            break;
        default:
            set_error("unknown layer op %d", op);
            return JPI_ERR_INVALID_ARG;
    }
    return check_launch("layer op (CUDA cores)");
}

// Step times are processed in groups of at most 8 so the shared-memory copy of the inputs
// stays at 8 x max(W, d_t) floats whatever the step count.
constexpr int TC_GROUP = 8;

// Modulation step times per pass of k_mod_gemv (its shared copy of X is MOD_GROUP x W floats).
constexpr int MOD_GROUP = 16;

template <typename T, int NG>
void launch_mod_gemv(jpi_handle* h, const float* X, float* Y, int R, cudaStream_t st) {
    const int W = h->W;
    int threads = (R / MOD_RT + h->num_sms - 1) / h->num_sms;   // about one CTA per SM
    threads = (threads + 31) / 32 * 32;
    threads = threads < 64 ? 64 : (threads > 256 ? 256 : threads);
    const int grid = (R + threads * MOD_RT - 1) / (threads * MOD_RT);
    k_mod_gemv<T, NG><<<grid, threads, sizeof(float) * NG * W, st>>>((const T*)h->mod_w, h->mod_b, X, Y, R, W);
}

// bf16 weights with the tensor-core path: the tcgen05 kernel of mod_tc.cu; otherwise (and for
// fp32 weights) the CUDA-core kernel above.
template <typename T>
jpi_status mod_gemv(jpi_handle* h, int g, const float* X, float* Y, int R, cudaStream_t st) {
    if (std::is_same<T, __nv_bfloat16>::value && h->mod_tc) return launch_mod_tc(h, X, Y, g, st);
    switch (g) {
#define JPI_MOD_CASE(n) case n: launch_mod_gemv<T, n>(h, X, Y, R, st); break;
        JPI_MOD_CASE(1) JPI_MOD_CASE(2) JPI_MOD_CASE(3) JPI_MOD_CASE(4) JPI_MOD_CASE(5) JPI_MOD_CASE(6)
        JPI_MOD_CASE(7) JPI_MOD_CASE(8) JPI_MOD_CASE(9) JPI_MOD_CASE(10) JPI_MOD_CASE(11)
        JPI_MOD_CASE(12) JPI_MOD_CASE(13) JPI_MOD_CASE(14) JPI_MOD_CASE(15) JPI_MOD_CASE(16)
#undef JPI_MOD_CASE
        default: break;
    }
    return JPI_OK;
}

template <typename T>
jpi_status set_mod_attrs(int smem) {
#define JPI_MOD_ATTR(n) \
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_mod_gemv<T, n>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    JPI_MOD_ATTR(1) JPI_MOD_ATTR(2) JPI_MOD_ATTR(3) JPI_MOD_ATTR(4) JPI_MOD_ATTR(5) JPI_MOD_ATTR(6)
    JPI_MOD_ATTR(7) JPI_MOD_ATTR(8) JPI_MOD_ATTR(9) JPI_MOD_ATTR(10) JPI_MOD_ATTR(11) JPI_MOD_ATTR(12)
    JPI_MOD_ATTR(13) JPI_MOD_ATTR(14) JPI_MOD_ATTR(15) JPI_MOD_ATTR(16)
#undef JPI_MOD_ATTR
    return JPI_OK;
}

template <typename T>
jpi_status time_cond(jpi_handle* h, int N, cudaStream_t st) {
    const int W = h->W, dt = h->dt;
    const int R = mod_rows(h->L) * W;
    const dim3 blk(256);
    for (int n0 = 0; n0 < N; n0 += TC_GROUP) {
        const int g = (N - n0) < TC_GROUP ? (N - n0) : TC_GROUP;
        k_gemv_multi<T, true><<<grid_for((long long)W * 32, 256, 1024), blk, sizeof(float) * g * dt, st>>>(
            (const T*)h->time_in_w, h->time_in_b, h->temb + (size_t)n0 * dt, h->c1 + (size_t)n0 * W, W, dt, g);
        k_gemv_multi<T, true><<<grid_for((long long)W * 32, 256, 1024), blk, sizeof(float) * g * W, st>>>(
            (const T*)h->time_out_w, h->time_out_b, h->c1 + (size_t)n0 * W, h->cond + (size_t)n0 * W, W, W, g);
    }
    for (int n0 = 0; n0 < N; n0 += MOD_GROUP) {
        const int g = (N - n0) < MOD_GROUP ? (N - n0) : MOD_GROUP;
        JPI_TRY(mod_gemv<T>(h, g, h->cond + (size_t)n0 * W, h->mods + (size_t)n0 * R, R, st));
    }
    return check_launch("time conditioning");
}

}  // namespace

jpi_status configure_simt_kernels(jpi_handle* h) {
    const int D = h->D, H = h->H;
    const int att_smem = (int)(sizeof(float) * ((size_t)H * D + 32 * (D + 1) + 32 * D));
    const int gemv_smem = (int)(sizeof(float) * (size_t)TC_GROUP * (h->W > h->dt ? h->W : h->dt));
    const int mod_smem = (int)(sizeof(float) * (size_t)MOD_GROUP * h->W);
    int dev = 0;
    JPI_CUDA_TRY(cudaGetDevice(&dev));
    JPI_CUDA_TRY(cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, dev));
    if (h->bf16) {
        using T = __nv_bfloat16;
        JPI_CUDA_TRY(cudaFuncSetAttribute(k_attn_simt<T, T, T>, cudaFuncAttributeMaxDynamicSharedMemorySize, att_smem));
        JPI_CUDA_TRY(cudaFuncSetAttribute(k_gemv_multi<T, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, gemv_smem));
        JPI_CUDA_TRY(cudaFuncSetAttribute(k_gemv_multi<T, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, gemv_smem));
        JPI_TRY(set_mod_attrs<T>(mod_smem));
    } else {
        using T = float;
        JPI_CUDA_TRY(cudaFuncSetAttribute(k_attn_simt<T, T, T>, cudaFuncAttributeMaxDynamicSharedMemorySize, att_smem));
        JPI_CUDA_TRY(cudaFuncSetAttribute(k_gemv_multi<T, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, gemv_smem));
        JPI_CUDA_TRY(cudaFuncSetAttribute(k_gemv_multi<T, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, gemv_smem));
        JPI_TRY(set_mod_attrs<float>(mod_smem));
    }
    return JPI_OK;
}

jpi_status launch_time_embed(jpi_handle* h, int nsteps, double t_override, cudaStream_t st) {
    k_time_embed<<<dim3(nsteps, (h->dt / 2 + 127) / 128), 128, 0, st>>>(h->temb, nsteps, h->dt, h->cfg.t_min_period,
                                                                      h->cfg.t_max_period, t_override);
    return check_launch("time embedding");
}

jpi_status launch_time_conditioning(jpi_handle* h, int nsteps, cudaStream_t st) {
    return h->bf16 ? time_cond<__nv_bfloat16>(h, nsteps, st) : time_cond<float>(h, nsteps, st);
}

// Time conditioning of one step time with caller-chosen scratch: sinusoid into temb [d_t],
// time-MLP hidden layer into c1 [W], conditioning vector into cond [W]; the modulation
// vectors go to the handle's step-0 slot, as with launch_time_conditioning(h, 1, ...).
jpi_status launch_time_conditioning_into(jpi_handle* h, double t, float* temb, float* c1,
                                         float* cond, cudaStream_t st) {
    const int W = h->W, dt = h->dt;
    const int R = mod_rows(h->L) * W;
    k_time_embed<<<dim3(1, (dt / 2 + 127) / 128), 128, 0, st>>>(temb, 1, dt, h->cfg.t_min_period, h->cfg.t_max_period, t);
    const dim3 blk(256);
    if (h->bf16) {
        using T = __nv_bfloat16;
        k_gemv_multi<T, true><<<grid_for((long long)W * 32, 256, 1024), blk, sizeof(float) * dt, st>>>(
            (const T*)h->time_in_w, h->time_in_b, temb, c1, W, dt, 1);
        k_gemv_multi<T, true><<<grid_for((long long)W * 32, 256, 1024), blk, sizeof(float) * W, st>>>(
            (const T*)h->time_out_w, h->time_out_b, c1, cond, W, W, 1);
        JPI_TRY(mod_gemv<T>(h, 1, cond, h->mods, R, st));
    } else {
        using T = float;
        k_gemv_multi<T, true><<<grid_for((long long)W * 32, 256, 1024), blk, sizeof(float) * dt, st>>>(
            (const T*)h->time_in_w, h->time_in_b, temb, c1, W, dt, 1);
        k_gemv_multi<T, true><<<grid_for((long long)W * 32, 256, 1024), blk, sizeof(float) * W, st>>>(
            (const T*)h->time_out_w, h->time_out_b, c1, cond, W, W, 1);
        JPI_TRY(mod_gemv<T>(h, 1, cond, h->mods, R, st));
    }
    return check_launch("time conditioning (caller scratch)");
}

jpi_status launch_embed(jpi_handle* h, int step, int B, int C, const float* x, cudaStream_t st) {
    const int S = C + h->n_ctx();
    // Scale and shift of layer 0's attention norm at this step.
    const float* ms = h->mods + (size_t)step * mod_rows(h->L) * h->W;
    launch_pdl(h, dim3((h->W + 127) / 128, B * S), dim3(128), 0, st, k_embed,
               h->h, h->tc ? (__nv_bfloat16*)h->hx : nullptr, ms, ms + h->W, h->tc ? h->ss : nullptr, h->maxMt,
               (const float*)h->state, x, (const float*)h->state_in_w, (const float*)h->state_in_b,
               (const float*)h->action_in_w, (const float*)h->action_in_b, (const float*)h->corr, h->n_ctx(), S, C,
               h->W, h->Sd, h->A);
    return check_launch("embed");
}

jpi_status launch_op_simt(jpi_handle* h, int op, int layer, int step, int B, int C,
                          cudaStream_t st) {
    return h->bf16 ? op_simt<__nv_bfloat16>(h, op, layer, step, B, C, st)
                   : op_simt<float>(h, op, layer, step, B, C, st);
}

jpi_status launch_layer_simt(jpi_handle* h, int layer, int step, int B, int C, cudaStream_t st) {
    for (int op = 2; op <= 6; ++op) JPI_TRY(launch_op_simt(h, op, layer, step, B, C, st));
    return JPI_OK;
}

jpi_status launch_final(jpi_handle* h, int step, int B, int C, float delta, float* x_inout,
                        float* v_out, float* out_copy, cudaStream_t st) {
    const int W = h->W;
    const float* ms = h->mods + (size_t)step * mod_rows(h->L) * W + (size_t)6 * h->L * W;
    launch_pdl(h, dim3(B * C), dim3(FIN_THREADS), sizeof(float) * W, st, k_final, (const float*)h->h, ms, ms + W,
               (const float*)h->action_out_w, (const float*)h->action_out_b, x_inout, v_out, out_copy,
               C + h->n_ctx(), h->n_ctx(), C, W, h->A, h->cfg.rms_eps, delta);
    return check_launch("final norm + Euler");
}

jpi_status launch_convert_kv(jpi_handle* h, const void* src, int src_fp32, void* dst, int B,
                             int P, cudaStream_t st) {
    const long long total = (long long)B * P * h->D;
    const int g = grid_for(total, 256, 8192);
    if (h->bf16) {
        if (src_fp32)
            k_convert_kv<float, __nv_bfloat16><<<g, 256, 0, st>>>((const float*)src, (__nv_bfloat16*)dst, P, h->D, h->kv_rows, total);
        else
            k_convert_kv<__nv_bfloat16, __nv_bfloat16><<<g, 256, 0, st>>>((const __nv_bfloat16*)src, (__nv_bfloat16*)dst, P, h->D, h->kv_rows, total);
    } else {
        if (src_fp32)
            k_convert_kv<float, float><<<g, 256, 0, st>>>((const float*)src, (float*)dst, P, h->D, h->kv_rows, total);
        else
            k_convert_kv<__nv_bfloat16, float><<<g, 256, 0, st>>>((const __nv_bfloat16*)src, (float*)dst, P, h->D, h->kv_rows, total);
    }
    return check_launch("prefix KV conversion");
}

}  // namespace jpi
