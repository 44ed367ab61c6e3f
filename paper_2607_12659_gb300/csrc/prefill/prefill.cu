// The VLM's LLM prefill (App. A, Tab. "Model architecture parameters of pi series VLA models",
// Sec. 4.3): Gemma-shaped blocks over the prefix tokens, writing each layer's rotated keys and
// values straight into the action expert's KV store.
//
// Every product here is a plain GEMM with batch * prefix rows (816 per request): the Q/K/V, output,
// gate/up and down projections, and per request the scores q K^T (all heads stacked as rows,
// since the single KV head is shared) and the probabilities times V. They run as bf16 cuBLASLt
// matmuls with fp32 accumulation; the residual stream stays fp32, the two residual projections
// accumulate into it in place (beta = 1). This file's own kernels do the rest: RMSNorm to a bf16
// operand, rotary coding of q and k from a table built once in double precision (with k and v
// scattered into the store), the row softmax, and GeGLU.
//
// Row-major products map onto cuBLASLt's column-major ones as Y^T = op(W) X^T: a row-major
// [rows][cols] buffer is the column-major [cols][rows] matrix with the same leading dimension.

#include <cublasLt.h>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <map>
#include <new>
#include <tuple>
#include <vector>

#include "jpi_prefill.h"

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

#define PF_LT(expr)                                                                                \
    do {                                                                                           \
        cublasStatus_t s_ = (expr);                                                                \
        if (s_ != CUBLAS_STATUS_SUCCESS)                                                           \
            return pfail(JPI_ERR_CUDA, "%s failed: %s (%s:%d)", #expr, cublasLtGetStatusString(s_), \
                         __FILE__, __LINE__);                                                      \
    } while (0)

#define PF_TRY(expr)                         \
    do {                                     \
        jpi_status s_ = (expr);              \
        if (s_ != JPI_OK) return s_;         \
    } while (0)

constexpr size_t WORKSPACE_BYTES = 32u << 20;

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

// y = h / sqrt(mean(h^2) + eps) * (1 + w), row by row; one warp per row (grid-stride).
template <typename TO>
__global__ void __launch_bounds__(256) k_pf_rmsnorm(const float* __restrict__ h, const float* __restrict__ w,
                                                    TO* __restrict__ y, long long rows, int W, float eps) {
    const int lane = threadIdx.x & 31;
    const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
    for (long long r = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < rows; r += nwarps) {
        const float* hr = h + r * W;
        float s = 0.f;
        for (int i = lane; i < W; i += 32) s = fmaf(hr[i], hr[i], s);
        const float rinv = 1.f / sqrtf(warp_sum(s) / (float)W + eps);
        TO* yr = y + r * W;
        for (int i = lane; i < W; i += 32) {
            const float v = hr[i] * rinv * (1.f + w[i]);
            if constexpr (sizeof(TO) == 2) yr[i] = __float2bfloat16_rn(v);
            else yr[i] = v;
        }
    }
}

// From the projections qkv [B P][(H + 2) D] (fp32): rotated queries q [B P][H][D] (bf16), and the
// rotated keys and the values of request b, row p into kd / vd + b stride + p D (bf16). One thread
// per (row, section, rotary pair); rope[p][j] = (cos, sin) of p base^(-2j/D).
__global__ void k_pf_rope_scatter(const float* __restrict__ qkv, const float2* __restrict__ rope,
                                  __nv_bfloat16* __restrict__ q, __nv_bfloat16* __restrict__ kd,
                                  __nv_bfloat16* __restrict__ vd, long long stride, int B, int P, int H,
                                  int D) {
    const int half = D / 2, secs = H + 2;
    const long long total = (long long)B * P * secs * half;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x) {
        const int j = (int)(idx % half);
        const int s = (int)((idx / half) % secs);
        const long long r = idx / ((long long)half * secs);   // b P + p
        const int p = (int)(r % P), b = (int)(r / P);
        const float* src = qkv + r * (long long)secs * D + (long long)s * D;
        float x1 = src[j], x2 = src[j + half];
        if (s <= H) {
            const float2 cs = rope[(size_t)p * half + j];
            const float r1 = x1 * cs.x - x2 * cs.y, r2 = x2 * cs.x + x1 * cs.y;
            x1 = r1;
            x2 = r2;
        }
        __nv_bfloat16* dst;
        if (s < H) dst = q + (r * H + s) * (long long)D;
        else dst = (s == H ? kd : vd) + b * stride + (long long)p * D;
        dst[j] = __float2bfloat16_rn(x1);
        dst[j + half] = __float2bfloat16_rn(x2);
    }
}

// probs[r][0 .. n) = softmax(s[r][0 .. n)) as bf16 (rows of stride ld); one warp per row.
__global__ void __launch_bounds__(256) k_pf_softmax(const float* __restrict__ s, __nv_bfloat16* __restrict__ p,
                                                    long long rows, int n, int ld) {
    const int lane = threadIdx.x & 31;
    const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
    for (long long r = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < rows; r += nwarps) {
        const float* sr = s + r * ld;
        float mx = -INFINITY;
        for (int j = lane; j < n; j += 32) mx = fmaxf(mx, sr[j]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        float den = 0.f;
        for (int j = lane; j < n; j += 32) den += expf(sr[j] - mx);
        const float inv = 1.f / warp_sum(den);
        __nv_bfloat16* pr = p + r * ld;
        for (int j = lane; j < n; j += 32) pr[j] = __float2bfloat16_rn(expf(sr[j] - mx) * inv);
    }
}

// z[r][j] = gelu_tanh(gu[r][j]) * gu[r][F + j] (gate rows first, then up rows, in the packed matrix).
__global__ void k_pf_geglu(const float* __restrict__ gu, __nv_bfloat16* __restrict__ z, long long rows, int F) {
    const long long total = rows * F;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x) {
        const long long r = idx / F;
        const int j = (int)(idx % F);
        const float* row = gu + r * 2 * (long long)F;
        z[idx] = __float2bfloat16_rn(gelu_tanh_f(row[j]) * row[F + j]);
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

struct GemmKey {
    int opw, M, N, K, ldx, ldw, ldy, tx, tw, ty, acc;
    unsigned alx, alw, aly;   // byte alignment of each operand's address (at most 256)
    bool operator<(const GemmKey& o) const {
        return std::tie(opw, M, N, K, ldx, ldw, ldy, tx, tw, ty, acc, alx, alw, aly) <
               std::tie(o.opw, o.M, o.N, o.K, o.ldx, o.ldw, o.ldy, o.tx, o.tw, o.ty, o.acc, o.alx, o.alw, o.aly);
    }
};

// Largest power of two up to 256 that divides the address.
unsigned alignment_of(const void* p) {
    const uintptr_t a = reinterpret_cast<uintptr_t>(p);
    unsigned r = 256;
    while (r > 1 && (a % r) != 0) r >>= 1;
    return r;
}

struct GemmPlan {
    cublasLtMatmulDesc_t desc = nullptr;
    cublasLtMatrixLayout_t a = nullptr, b = nullptr, c = nullptr;
    cublasLtMatmulAlgo_t algo;
};

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
    __nv_bfloat16* xn = nullptr;     // [Bm Pm][max(W, F)] GEMM operand (normed h, or z)
    float* qkv = nullptr;            // [Bm Pm][(H + 2) D]
    __nv_bfloat16* q = nullptr;      // [Bm Pm][H][D]
    __nv_bfloat16* o = nullptr;      // [Bm Pm][H D]
    float* gu = nullptr;             // [Bm Pm][2 F]
    float* sc = nullptr;             // [H Pm][Pp] scores of one request
    __nv_bfloat16* pr = nullptr;     // [H Pm][Pp] probabilities of one request
    void* ws = nullptr;
    cublasLtHandle_t lt = nullptr;
    std::map<GemmKey, GemmPlan> plans;
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

void destroy_plan(GemmPlan& pl) {
    if (pl.desc) cublasLtMatmulDescDestroy(pl.desc);
    if (pl.a) cublasLtMatrixLayoutDestroy(pl.a);
    if (pl.b) cublasLtMatrixLayoutDestroy(pl.b);
    if (pl.c) cublasLtMatrixLayoutDestroy(pl.c);
    pl = GemmPlan();
}

void release(jpi_prefill_handle* h) {
    for (auto& kv : h->plans) destroy_plan(kv.second);
    h->plans.clear();
    if (h->lt) cublasLtDestroy(h->lt);
    h->lt = nullptr;
    for (void* p : h->allocs) cudaFree(p);
    h->allocs.clear();
}

// Descriptors, layouts and the heuristic's algorithm for one product shape; the algorithm is
// chosen for the operands' actual address alignment (cuBLASLt otherwise assumes 256 bytes).
cublasStatus_t make_plan(jpi_prefill_handle* h, const GemmKey& k, GemmPlan* pl) {
    cublasStatus_t s = cublasLtMatmulDescCreate(&pl->desc, CUBLAS_COMPUTE_32F, CUDA_R_32F);
    const cublasOperation_t opa = k.opw ? CUBLAS_OP_T : CUBLAS_OP_N, opb = CUBLAS_OP_N;
    if (s == CUBLAS_STATUS_SUCCESS)
        s = cublasLtMatmulDescSetAttribute(pl->desc, CUBLASLT_MATMUL_DESC_TRANSA, &opa, sizeof(opa));
    if (s == CUBLAS_STATUS_SUCCESS)
        s = cublasLtMatmulDescSetAttribute(pl->desc, CUBLASLT_MATMUL_DESC_TRANSB, &opb, sizeof(opb));
    if (s == CUBLAS_STATUS_SUCCESS)
        s = k.opw ? cublasLtMatrixLayoutCreate(&pl->a, (cudaDataType)k.tw, (uint64_t)k.K, (uint64_t)k.N, (int64_t)k.ldw)
                  : cublasLtMatrixLayoutCreate(&pl->a, (cudaDataType)k.tw, (uint64_t)k.N, (uint64_t)k.K, (int64_t)k.ldw);
    if (s == CUBLAS_STATUS_SUCCESS)
        s = cublasLtMatrixLayoutCreate(&pl->b, (cudaDataType)k.tx, (uint64_t)k.K, (uint64_t)k.M, (int64_t)k.ldx);
    if (s == CUBLAS_STATUS_SUCCESS)
        s = cublasLtMatrixLayoutCreate(&pl->c, (cudaDataType)k.ty, (uint64_t)k.N, (uint64_t)k.M, (int64_t)k.ldy);
    if (s != CUBLAS_STATUS_SUCCESS) return s;
    cublasLtMatmulPreference_t pref = nullptr;
    s = cublasLtMatmulPreferenceCreate(&pref);
    if (s != CUBLAS_STATUS_SUCCESS) return s;
    const uint64_t wsb = WORKSPACE_BYTES;
    const uint32_t al[4] = {k.alw, k.alx, k.aly, k.aly};   // A = W, B = X, C = D = Y
    s = cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MAX_WORKSPACE_BYTES, &wsb, sizeof(wsb));
    if (s == CUBLAS_STATUS_SUCCESS)
        s = cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MIN_ALIGNMENT_A_BYTES, &al[0], sizeof(al[0]));
    if (s == CUBLAS_STATUS_SUCCESS)
        s = cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MIN_ALIGNMENT_B_BYTES, &al[1], sizeof(al[1]));
    if (s == CUBLAS_STATUS_SUCCESS)
        s = cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MIN_ALIGNMENT_C_BYTES, &al[2], sizeof(al[2]));
    if (s == CUBLAS_STATUS_SUCCESS)
        s = cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MIN_ALIGNMENT_D_BYTES, &al[3], sizeof(al[3]));
    cublasLtMatmulHeuristicResult_t res;
    int nres = 0;
    if (s == CUBLAS_STATUS_SUCCESS)
        s = cublasLtMatmulAlgoGetHeuristic(h->lt, pl->desc, pl->a, pl->b, pl->c, pl->c, pref, 1, &res, &nres);
    cublasLtMatmulPreferenceDestroy(pref);
    if (s == CUBLAS_STATUS_SUCCESS && nres < 1) s = CUBLAS_STATUS_NOT_SUPPORTED;
    if (s == CUBLAS_STATUS_SUCCESS) pl->algo = res.algo;
    return s;
}

// Y [M][N] (row-major, leading dimension ldy) = alpha X [M][K] op(W) + beta Y, where op(W) = W^T
// for W stored [N][K] (w_nk) and W for W stored [K][N]. As a column-major product:
// Y^T (N x M) = op_A(A) (N x K) * X^T (K x M) with A the W buffer (column-major K x N, transposed,
// when w_nk; column-major N x K otherwise) and X^T the X buffer as column-major K x M.
jpi_status row_gemm(jpi_prefill_handle* h, cudaStream_t st, const void* X, cudaDataType tx, int ldx,
                    const void* Wm, cudaDataType tw, int ldw, bool w_nk, void* Y, cudaDataType ty, int ldy,
                    int M, int N, int K, float alpha, float beta) {
    const GemmKey key{w_nk ? 1 : 0, M, N, K, ldx, ldw, ldy, (int)tx, (int)tw, (int)ty, beta != 0.f ? 1 : 0,
                      alignment_of(X), alignment_of(Wm), alignment_of(Y)};
    auto it = h->plans.find(key);
    if (it == h->plans.end()) {
        GemmPlan pl;
        const cublasStatus_t s = make_plan(h, key, &pl);
        if (s != CUBLAS_STATUS_SUCCESS) {
            destroy_plan(pl);
            return pfail(JPI_ERR_UNSUPPORTED, "no cuBLASLt algorithm for a %d x %d x %d product (%s)", M, N, K,
                         cublasLtGetStatusString(s));
        }
        it = h->plans.emplace(key, pl).first;
    }
    const GemmPlan& pl = it->second;
    PF_LT(cublasLtMatmul(h->lt, pl.desc, &alpha, Wm, pl.a, X, pl.b, &beta, Y, pl.c, Y, pl.c, &pl.algo, h->ws,
                         WORKSPACE_BYTES, st));
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
    const bool dev = w->on_device != 0;
    if (!w->attn_norm || !w->wq || !w->wk || !w->wv || !w->wo || !w->mlp_norm || !w->w_gate || !w->w_up ||
        !w->w_down || !w->final_norm)
        return pfail(JPI_ERR_INVALID_ARG, "a weight array is NULL");

    PF_LT(cublasLtCreate(&h->lt));
    char* ws = nullptr;
    PF_TRY(pf_alloc(h, &ws, WORKSPACE_BYTES));
    h->ws = ws;
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
        PF_TRY(pf_alloc(h, &lw.wgu, 2 * F * W));
        PF_TRY(put_bf16(h, dev, staging, lw.wgu, w->w_gate[l], F * W, "w_gate", l));
        PF_TRY(put_bf16(h, dev, staging, lw.wgu + F * W, w->w_up[l], F * W, "w_up", l));
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
    PF_TRY(pf_alloc(h, &h->xn, Mm * (W > F ? W : F)));
    PF_TRY(pf_alloc(h, &h->qkv, Mm * (size_t)h->QKV));
    PF_TRY(pf_alloc(h, &h->q, Mm * HD));
    PF_TRY(pf_alloc(h, &h->o, Mm * HD));
    PF_TRY(pf_alloc(h, &h->gu, Mm * 2 * F));
    PF_TRY(pf_alloc(h, &h->sc, (size_t)h->H * h->Pm * h->Pp));
    PF_TRY(pf_alloc(h, &h->pr, (size_t)h->H * h->Pm * h->Pp));
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
    const cudaDataType BF = CUDA_R_16BF, F32 = CUDA_R_32F;

    k_pf_load_x<<<grid_for(M * W), 256, 0, st>>>(x, x_is_fp32, h->h, M * W);
    PF_CUDA(cudaGetLastError());
    for (int l = 0; l < h->L; ++l) {
        const LayerW& lw = h->layers[(size_t)l];
        __nv_bfloat16* kd = static_cast<__nv_bfloat16*>(k_layers[l]);
        __nv_bfloat16* vd = static_cast<__nv_bfloat16*>(v_layers[l]);
        // Attention sublayer.
        k_pf_rmsnorm<__nv_bfloat16><<<grid_for(M * 32), 256, 0, st>>>(h->h, lw.attn_norm, h->xn, M, W, eps);
        PF_CUDA(cudaGetLastError());
        PF_TRY(row_gemm(h, st, h->xn, BF, W, lw.wqkv, BF, W, true, h->qkv, F32, h->QKV, (int)M, h->QKV, W, 1.f, 0.f));
        k_pf_rope_scatter<<<grid_for(M * (H + 2) * (D / 2)), 256, 0, st>>>(h->qkv, h->rope, h->q, kd, vd,
                                                                             request_stride, batch, P, H, D);
        PF_CUDA(cudaGetLastError());
        for (int b = 0; b < batch; ++b) {
            const __nv_bfloat16* qb = h->q + (size_t)b * P * H * D;     // [(P H)][D]
            const __nv_bfloat16* kb = kd + (size_t)b * request_stride;  // [P][D]
            const __nv_bfloat16* vb = vd + (size_t)b * request_stride;  // [P][D]
            __nv_bfloat16* ob = h->o + (size_t)b * P * H * D;           // [(P H)][D] = [P][H D]
            PF_TRY(row_gemm(h, st, qb, BF, D, kb, BF, D, true, h->sc, F32, Pp, P * H, P, D, scale, 0.f));
            k_pf_softmax<<<grid_for((long long)P * H * 32), 256, 0, st>>>(h->sc, h->pr, (long long)P * H, P, Pp);
            PF_CUDA(cudaGetLastError());
            PF_TRY(row_gemm(h, st, h->pr, BF, Pp, vb, BF, D, false, ob, BF, D, P * H, D, P, 1.f, 0.f));
        }
        PF_TRY(row_gemm(h, st, h->o, BF, H * D, lw.wo, BF, H * D, true, h->h, F32, W, (int)M, W, H * D, 1.f, 1.f));
        // MLP sublayer.
        k_pf_rmsnorm<__nv_bfloat16><<<grid_for(M * 32), 256, 0, st>>>(h->h, lw.mlp_norm, h->xn, M, W, eps);
        PF_CUDA(cudaGetLastError());
        PF_TRY(row_gemm(h, st, h->xn, BF, W, lw.wgu, BF, W, true, h->gu, F32, 2 * F, (int)M, 2 * F, W, 1.f, 0.f));
        k_pf_geglu<<<grid_for(M * F), 256, 0, st>>>(h->gu, h->xn, M, F);
        PF_CUDA(cudaGetLastError());
        PF_TRY(row_gemm(h, st, h->xn, BF, F, lw.wd, BF, F, true, h->h, F32, W, (int)M, W, F, 1.f, 1.f));
    }
    if (out_final) {
        k_pf_rmsnorm<float><<<grid_for(M * 32), 256, 0, st>>>(h->h, h->final_norm, out_final, M, W, eps);
        PF_CUDA(cudaGetLastError());
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
