// Tensor-core path of the bf16 expert layers: tcgen05 GEMMs fed by bulk tensor copies.
//
// Every projection of a layer is a skinny GEMM Y[tokens][out] = X[tokens][K] W[out][K]^T with
// tokens = batch x (chunk + 1) (51 at batch 1). It runs "swap-AB": a 128-row tile of W is the
// A operand (M = 128), a 64-token tile of X is the B operand (N = 64), and the fp32 product
// sits in TMEM. The K dimension of each weight tile is split across the CTAs of one thread-
// block cluster. Each CTA loads its weight blocks with bulk tensor copies before it waits on
// the previous kernel (weights do not depend on it); after the wait it loads its X blocks the
// same way from the bf16 activation the previous op left in global memory (for the two
// RMSNorm-fed projections it then applies the norm and the time-conditioned scale/shift in
// shared memory), multiplies, and the cluster reduces its fp32 partials through distributed
// shared memory in a fixed rank order, so results do not depend on timing. Each CTA applies
// the epilogue to its slice of the reduced tile: rotary encoding + scatter into the query
// buffer and KV store (QKV), GeGLU (gate/up), or the gated residual update of the fp32 stream
// with its bf16 copy and per-token sums of squares for the next RMSNorm (O, down).

#include "tc_path.h"
#include "ptx.h"

#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <type_traits>
#include <cmath>
#include <cstdlib>
#include <vector>

namespace jpi {
namespace {

constexpr int NT = 64;                         // tokens per MMA (N)
constexpr int TILE_ROWS = 128;                 // weight rows per tile (M)
constexpr int KBLK = 64;                       // K elements per block: one 128-byte swizzle row
constexpr int TILE_BYTES = TILE_ROWS * KBLK * 2;
constexpr int XBLK_BYTES = NT * KBLK * 2;
constexpr int PART_BYTES = TILE_ROWS * NT * 2;  // fp16 partial of one tile (128-byte rows)
constexpr int GEMM_THREADS = 256;
constexpr int QUADS = NT / 4;                  // token quads per tile
constexpr uint64_t WAIT_LIMIT_NS = 200ull * 1000 * 1000;   // 0.2 s

enum GemmKind { G_QKV = 0, G_O = 1, G_GU = 2, G_DOWN = 3 };

struct GemmArgs {
    int Mt, K, nkb, kpb, splits;
    int ntiles;              // weight tiles (large-M kernel: tiles walked by the persistent CTAs)
    // RMSNorm-fed projections (QKV, gate/up): W u = rinv * (W xs) + W beta, with xs = (1 + sigma) h
    // and beta packed as tiles of 63 tokens + 1 beta row by the producer of h, and rinv from the
    // per-token sums of squares it left.
    const float* ss;         // [nslot][ss_ld]: sums of h^2 over disjoint feature ranges
    int nslot, ss_ld;
    float eps, inv_w;
    // Gated residual epilogue (O, down).
    float* hres;
    __nv_bfloat16* xs;       // operand of the next norm-fed GEMM (null: none follows)
    const float* sigma_next; // that norm's scale and shift
    const float* beta_next;
    const float* gamma;
    float* ss_out;           // slot (tile * splits + rank): this CTA's features
    int W;
    // QKV epilogue.
    __nv_bfloat16* q;
    __nv_bfloat16* kst;
    __nv_bfloat16* vst;
    const float2* rope;
    int S, H, D, P, kv_rows;
    // GeGLU epilogue.
    __nv_bfloat16* z;
    int F;
    int* err;
};

// GELU, tanh form, with the hardware tanh (PTX tanh.approx.f32, relative error about 2^-11): the
// product it enters is rounded to bf16 (2^-9) right after, and the fp32 verification mode runs the
// CUDA-core kernels with the library tanh.
__device__ __forceinline__ float gelu_tanh(float y) {
    const float k0 = 0.7978845608028654f;   // sqrt(2 / pi)
    float th;
    asm("tanh.approx.f32 %0, %1;" : "=f"(th) : "f"(k0 * (y + 0.044715f * y * y * y)));
    return 0.5f * y * (1.f + th);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ float2 unpack_half2(uint32_t v) {
    __half2 b = *reinterpret_cast<__half2*>(&v);
    return __half22float2(b);
}

__device__ __forceinline__ void set_device_error(int* err, int code) { atomicCAS(err, 0, code); }

__device__ __forceinline__ float f4get(const float4& v, int e) {
    return e == 0 ? v.x : e == 1 ? v.y : e == 2 ? v.z : v.w;
}
__device__ __forceinline__ float4 half4_to_float4(uint2 v) {
    const float2 lo = __half22float2(*reinterpret_cast<__half2*>(&v.x));
    const float2 hi = __half22float2(*reinterpret_cast<__half2*>(&v.y));
    return make_float4(lo.x, lo.y, hi.x, hi.y);
}
__device__ __forceinline__ void f4add(float4& a, const float4& b) {
    a.x += b.x;
    a.y += b.y;
    a.z += b.z;
    a.w += b.w;
}

// Shared-memory layout of one GEMM CTA (byte offsets from the 1024-aligned base).
struct GemmSmem {
    int x, recv, misc, ssred, bars, total;
};
__host__ __device__ __forceinline__ GemmSmem gemm_layout(int kpb, int splits, bool norm_in) {
    GemmSmem L;
    const int xbytes = kpb * XBLK_BYTES > PART_BYTES ? kpb * XBLK_BYTES : PART_BYTES;
    const int ssred_bytes = 2 * NT * (int)sizeof(float);
    L.x = kpb * TILE_BYTES;
    L.recv = L.x + xbytes;
    L.misc = L.recv + (splits - 1) * (TILE_ROWS / splits) * NT * 2;
    int end = L.misc + (norm_in ? 4 * NT * (int)sizeof(float) : 0);   // ss partials + rinv
    if (norm_in) {
        L.ssred = L.misc;                               // unused by the norm-fed kinds
    } else if (xbytes >= PART_BYTES + ssred_bytes) {
        L.ssred = L.x + PART_BYTES;                     // X blocks are dead once the MMA is done
    } else {
        L.ssred = end;
        end += ssred_bytes;
    }
    L.bars = (end + 7) & ~7;
    L.total = L.bars + 64;   // 4 mbarriers, the TMEM address, the error flag
    return L;
}

#include "gemm_kernel.cuh"
#include "gemm_big.cuh"

// ---------------------------------------------------------------------------------------------
// Host side: packing, plans, tensor maps, launches.

size_t gemm_smem(int kpb, int splits, bool norm_in) {
    return 1024 + (size_t)gemm_layout(kpb, splits, norm_in).total;
}

// Chooses the K blocks per CTA: one wave on the device, then at most 8 CTAs per cluster (each
// extra rank adds two pushes to every CTA's exchange and a slice to every owner's sum, which
// measured slower than streaming more weight per CTA), then little weight per SM, then shared
// memory small enough (<= 113 KB) for two CTAs per SM.
bool make_plan(int rows, int K, int max_cluster, int num_sms, bool norm_in, GemmPlan* out) {
    if (rows % TILE_ROWS || K % KBLK) return false;
    GemmPlan best;
    long best_score = -1;
    const int ntiles = rows / TILE_ROWS, nkb = K / KBLK;
    for (int kpb = 1; kpb <= 8; kpb *= 2) {
        if (nkb % kpb) continue;
        const int splits = nkb / kpb;
        if (splits > std::min(max_cluster, MAX_SPLIT_K) || 64 % splits) continue;
        const size_t smem = gemm_smem(kpb, splits, norm_in);
        if (smem > 227 * 1024) continue;
        const int res = std::min(2, (int)((228 * 1024) / (smem + 1024)));
        const int ctas = ntiles * splits;
        const long waves = (ctas + (long)num_sms * res - 1) / ((long)num_sms * res);
        const long per_sm = (ctas + num_sms - 1) / num_sms;
        const long score = waves * 10000 + std::max(splits - 8, 0) * 100 + per_sm * kpb * 10 +
                           (smem > 113 * 1024 ? 5 : 0) + (ctas > num_sms ? 1 : 0);
        if (best_score < 0 || score < best_score) {
            best_score = score;
            best.rows = rows; best.K = K; best.ntiles = ntiles; best.nkb = nkb; best.kpb = kpb;
            best.splits = splits; best.ctas = ctas; best.smem = smem;
        }
    }
    if (best_score < 0) return false;
    *out = best;
    return true;
}

// fp32 [rows][K] -> bf16 tiles; source row s lands on tiled row dest_row[s] (identity if null).
__global__ void k_pack_tiles(const float* __restrict__ src, __nv_bfloat16* __restrict__ dst,
                             const int* __restrict__ dest_row, int rows, int K) {
    const int nkb = K / KBLK;
    const long long total = (long long)rows * K;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int s = (int)(i / K), k = (int)(i % K);
        const int R = dest_row ? dest_row[s] : s;
        const size_t o = ((size_t)(R / TILE_ROWS) * nkb + k / KBLK) * (TILE_ROWS * KBLK) +
                         (size_t)(R % TILE_ROWS) * KBLK + (k % KBLK);
        dst[o] = __float2bfloat16_rn(src[i]);
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

// 2D 16-bit tensor map over [rows][cols] (row-major), 128-byte swizzle, box {64 cols, box_rows}.
jpi_status make_tmap(const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows, CUtensorMap* map,
                     CUtensorMapDataType dtype = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16) {
    auto enc = get_encode();
    if (!enc) {
        set_error("cuTensorMapEncodeTiled is unavailable from the driver");
        return JPI_ERR_CUDA;
    }
    const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    const cuuint32_t box[2] = {(cuuint32_t)KBLK, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, dtype, 2, (void*)base, dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        set_error("cuTensorMapEncodeTiled failed (%d)", (int)r);
        return JPI_ERR_CUDA;
    }
    return JPI_OK;
}

template <typename T>
jpi_status tc_alloc(jpi_handle* h, T** p, size_t count) {
    void* q = nullptr;
    if (cudaMalloc(&q, count * sizeof(T)) != cudaSuccess) {
        cudaGetLastError();
        set_error("cudaMalloc of %zu bytes failed", count * sizeof(T));
        return JPI_ERR_OOM;
    }
    h->allocations.push_back(q);
    h->device_bytes += count * sizeof(T);
    *p = (T*)q;
    return JPI_OK;
}

// Puts one fp32 tensor (host or device) into device memory at `dst` (fp32).
jpi_status stage(float* dst, const float* src, size_t n, bool on_device) {
    if (!src) {
        set_error("a per-layer weight tensor is NULL");
        return JPI_ERR_INVALID_ARG;
    }
    JPI_CUDA_TRY(cudaMemcpy(dst, src, n * sizeof(float),
                            on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice));
    return JPI_OK;
}

jpi_status pack(const float* tmp, __nv_bfloat16* dst, const int* dmap, int rows, int K) {
    const long long total = (long long)rows * K;
    const int g = (int)std::min<long long>((total + 255) / 256, 16384);
    k_pack_tiles<<<g, 256>>>(tmp, dst, dmap, rows, K);
    JPI_CUDA_TRY(cudaGetLastError());
    return JPI_OK;
}

template <int KIND>
jpi_status launch_gemm(jpi_handle* h, const GemmPlan& pl, const CUtensorMap& wmap,
                       const CUtensorMap& xmap, const GemmArgs& a, cudaStream_t st) {
    // One grid row per token tile (63 tokens + the beta row for the norm-fed kinds, else 64).
    constexpr int TT = (KIND == G_QKV || KIND == G_GU) ? XS_TOKENS : NT;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(pl.ctas, (unsigned)std::max(1, (a.Mt + TT - 1) / TT));
    cfg.blockDim = dim3(GEMM_THREADS);
    cfg.dynamicSmemBytes = pl.smem;
    cfg.stream = st;
    cudaLaunchAttribute attrs[2];
    int n = 0;
    attrs[n].id = cudaLaunchAttributeClusterDimension;
    attrs[n].val.clusterDim.x = pl.splits;
    attrs[n].val.clusterDim.y = 1;
    attrs[n].val.clusterDim.z = 1;
    ++n;
    if (h->pdl) {
        attrs[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attrs[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    cfg.attrs = attrs;
    cfg.numAttrs = n;
    cudaError_t e = cudaLaunchKernelEx(&cfg, k_tc_gemm<KIND>, wmap, xmap, a);
    if (e != cudaSuccess) {
        set_error("tensor-core GEMM launch failed: %s", cudaGetErrorString(e));
        return JPI_ERR_CUDA;
    }
    return JPI_OK;
}

// Large-M variant: persistent CTAs over (weight tile, 128-row operand tile) units. The residual
// kinds (few weight tiles, long K) may split each unit's K range over a cluster of S CTAs so that
// the units fill the GPU: S is the one of 1, 2, 4, 8 with the fewest estimated K blocks per SM,
// counting waves of S x units CTAs and an exchange worth BIG_SPLIT_COST K blocks for S > 1.
constexpr int BIG_SPLIT_COST = 4;

// Clusters of S large-M CTAs that can run at once (one CTA per SM; clusters of 8 leave some SMs
// of each GPC idle), from the occupancy query at prepare time.
int big_clusters(const jpi_handle* h, int S) {
    const int i = S == 1 ? 0 : S == 2 ? 1 : S == 4 ? 2 : 3;
    return h->big_clusters[i] > 0 ? h->big_clusters[i] : h->num_sms / S;
}

int big_split(const jpi_handle* h, int kind, int units, int nkb) {
    if (kind != G_O && kind != G_DOWN) return 1;
    if (h->big_split > 0) return nkb % h->big_split == 0 ? h->big_split : 1;
    int best = 1;
    long best_cost = -1;
    for (int S = 1; S <= 8; S *= 2) {
        if (nkb % S || nkb / S < 2) continue;
        const long waves = (units + big_clusters(h, S) - 1) / big_clusters(h, S);
        const long cost = waves * (nkb / S + (S > 1 ? BIG_SPLIT_COST : 0));
        if (best_cost < 0 || cost < best_cost) {
            best_cost = cost;
            best = S;
        }
    }
    return best;
}

template <int KIND, int S>
jpi_status launch_big_s(jpi_handle* h, int units, const CUtensorMap& wmap, const CUtensorMap& xmap,
                        const GemmArgs& a, cudaStream_t st) {
    cudaLaunchConfig_t cfg = {};
    // Persistent: one CTA per SM (clusters of S that all run at once, at most one per unit).
    cfg.gridDim = dim3((unsigned)(S * std::min(units, big_clusters(h, S))));
    cfg.blockDim = dim3(BIG_THREADS);
    cfg.dynamicSmemBytes = 1024 + big_smem_bytes<S>();
    cfg.stream = st;
    cudaLaunchAttribute attrs[2];
    int n = 0;
    if (S > 1) {
        attrs[n].id = cudaLaunchAttributeClusterDimension;
        attrs[n].val.clusterDim.x = S;
        attrs[n].val.clusterDim.y = 1;
        attrs[n].val.clusterDim.z = 1;
        ++n;
    }
    if (h->pdl) {
        attrs[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attrs[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    cfg.attrs = attrs;
    cfg.numAttrs = n;
    cudaError_t e = cudaLaunchKernelEx(&cfg, k_tc_gemm_big<KIND, S>, wmap, xmap, a);
    if (e != cudaSuccess) {
        set_error("tensor-core GEMM launch failed: %s", cudaGetErrorString(e));
        return JPI_ERR_CUDA;
    }
    return JPI_OK;
}

template <int KIND>
jpi_status launch_gemm_big(jpi_handle* h, const GemmPlan& pl, const CUtensorMap& wmap,
                           const CUtensorMap& xmap, const GemmArgs& a, cudaStream_t st) {
    constexpr int TT = (KIND == G_QKV || KIND == G_GU) ? 2 * XS_TOKENS : BIG_NT;
    const int units = pl.ntiles * std::max(1, (a.Mt + TT - 1) / TT);
    GemmArgs ab = a;
    ab.ntiles = pl.ntiles;
    if constexpr (KIND == G_O || KIND == G_DOWN) {
        switch (big_split(h, KIND, units, pl.nkb)) {
            case 2: return launch_big_s<KIND, 2>(h, units, wmap, xmap, ab, st);
            case 4: return launch_big_s<KIND, 4>(h, units, wmap, xmap, ab, st);
            case 8: return launch_big_s<KIND, 8>(h, units, wmap, xmap, ab, st);
            default: break;
        }
    }
    return launch_big_s<KIND, 1>(h, units, wmap, xmap, ab, st);
}

GemmArgs base_args(jpi_handle* h, int B, int C, const GemmPlan& pl) {
    GemmArgs a = {};
    a.Mt = B * (C + h->n_ctx());
    a.K = pl.K;
    a.nkb = pl.nkb;
    a.kpb = pl.kpb;
    a.splits = pl.splits;
    a.ss = h->ss;
    a.nslot = h->W / TILE_ROWS;
    a.ss_ld = h->maxMt;
    a.eps = h->cfg.rms_eps;
    a.inv_w = 1.f / (float)h->W;
    a.W = h->W;
    a.S = C + h->n_ctx();
    a.H = h->H;
    a.D = h->D;
    a.P = h->cur_prefix;
    a.kv_rows = h->kv_rows;
    a.F = h->F;
    a.err = h->dev_err;
    return a;
}

}  // namespace

jpi_status tc_make_tmap(const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows, CUtensorMap* map) {
    return make_tmap(base, rows, cols, box_rows, map);
}

bool tc_supported(const jpi_handle* h) {
    return h->W % TILE_ROWS == 0 && h->D % TILE_ROWS == 0 && h->F % 64 == 0 && h->HD % KBLK == 0 &&
           h->W / TILE_ROWS <= 64;
}

jpi_status tc_pack_layers(jpi_handle* h, const jpi_weights* w, float* tmp, bool on_device) {
    const int W = h->W, D = h->D, F = h->F, HD = h->HD, QKV = h->QKV;
    // Tiled row of every source row: QKV pairs (d, d + D/2) of each head section share a tile
    // (rows r and r + 64); gate row f and up row f share tile f / 64.
    std::vector<int> qmap(QKV), gmap(F), umap(F);
    const int hd = D / 2;
    for (int s = 0; s < QKV; ++s) {
        const int sec = s / D, dd = s % D, half = dd / hd, d = dd % hd;
        const int pair = sec * hd + d;
        qmap[s] = (pair / 64) * TILE_ROWS + half * 64 + pair % 64;
    }
    for (int f = 0; f < F; ++f) {
        gmap[f] = (f / 64) * TILE_ROWS + f % 64;
        umap[f] = (f / 64) * TILE_ROWS + 64 + f % 64;
    }
    int* dmaps = nullptr;
    JPI_TRY(tc_alloc(h, &dmaps, (size_t)QKV + 2 * F));
    JPI_CUDA_TRY(cudaMemcpy(dmaps, qmap.data(), QKV * sizeof(int), cudaMemcpyHostToDevice));
    JPI_CUDA_TRY(cudaMemcpy(dmaps + QKV, gmap.data(), F * sizeof(int), cudaMemcpyHostToDevice));
    JPI_CUDA_TRY(cudaMemcpy(dmaps + QKV + F, umap.data(), F * sizeof(int), cudaMemcpyHostToDevice));

    h->tiled.resize(h->L);
    for (int l = 0; l < h->L; ++l) {
        LayerTiled& t = h->tiled[l];
        JPI_TRY(tc_alloc(h, &t.qkv, (size_t)QKV * W));
        JPI_TRY(tc_alloc(h, &t.o, (size_t)W * HD));
        JPI_TRY(tc_alloc(h, &t.gu, (size_t)2 * F * W));
        JPI_TRY(tc_alloc(h, &t.down, (size_t)W * F));
        JPI_TRY(stage(tmp, w->wq[l], (size_t)HD * W, on_device));
        JPI_TRY(stage(tmp + (size_t)HD * W, w->wk[l], (size_t)D * W, on_device));
        JPI_TRY(stage(tmp + (size_t)(HD + D) * W, w->wv[l], (size_t)D * W, on_device));
        JPI_TRY(pack(tmp, t.qkv, dmaps, QKV, W));
        JPI_TRY(stage(tmp, w->wo[l], (size_t)W * HD, on_device));
        JPI_TRY(pack(tmp, t.o, nullptr, W, HD));
        JPI_TRY(stage(tmp, w->w_gate[l], (size_t)F * W, on_device));
        JPI_TRY(pack(tmp, t.gu, dmaps + QKV, F, W));
        JPI_TRY(stage(tmp, w->w_up[l], (size_t)F * W, on_device));
        JPI_TRY(pack(tmp, t.gu, dmaps + QKV + F, F, W));
        JPI_TRY(stage(tmp, w->w_down[l], (size_t)W * F, on_device));
        JPI_TRY(pack(tmp, t.down, nullptr, W, F));
    }
    JPI_CUDA_TRY(cudaDeviceSynchronize());
    return JPI_OK;
}

jpi_status tc_prepare(jpi_handle* h) {
    int dev = 0, sms = 0;
    JPI_CUDA_TRY(cudaGetDevice(&dev));
    JPI_CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    h->num_sms = sms;
    if (attn_tc_supported(h)) JPI_TRY(attn_tc_prepare(h));
    JPI_TRY(attn_t5_prepare(h));
    const char* pdl_env = std::getenv("JPI_PDL");
    h->pdl = !(pdl_env && pdl_env[0] == '0');

    int max_cluster = 16;
    auto kernels = {k_tc_gemm<G_QKV>, k_tc_gemm<G_O>, k_tc_gemm<G_GU>, k_tc_gemm<G_DOWN>};
    for (auto k : kernels) {
        if (cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
            cudaGetLastError();
            max_cluster = 8;
        }
        JPI_CUDA_TRY(cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024));
    }
    auto big1 = {k_tc_gemm_big<G_QKV, 1>, k_tc_gemm_big<G_O, 1>, k_tc_gemm_big<G_GU, 1>, k_tc_gemm_big<G_DOWN, 1>};
    for (auto k : big1)
        JPI_CUDA_TRY(cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, 1024 + big_smem_bytes<1>()));
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_tc_gemm_big<G_O, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize, 1024 + big_smem_bytes<2>()));
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_tc_gemm_big<G_DOWN, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize, 1024 + big_smem_bytes<2>()));
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_tc_gemm_big<G_O, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize, 1024 + big_smem_bytes<4>()));
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_tc_gemm_big<G_DOWN, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize, 1024 + big_smem_bytes<4>()));
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_tc_gemm_big<G_O, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize, 1024 + big_smem_bytes<8>()));
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_tc_gemm_big<G_DOWN, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize, 1024 + big_smem_bytes<8>()));
    {
        auto query = [&](const void* fn, int S, int smem) {
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3((unsigned)(S * (sms / S)));
            cfg.blockDim = dim3(BIG_THREADS);
            cfg.dynamicSmemBytes = (size_t)smem;
            cudaLaunchAttribute at;
            at.id = cudaLaunchAttributeClusterDimension;
            at.val.clusterDim.x = S;
            at.val.clusterDim.y = 1;
            at.val.clusterDim.z = 1;
            cfg.attrs = &at;
            cfg.numAttrs = 1;
            int n = 0;
            if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess) {
                cudaGetLastError();
                n = 0;
            }
            return n;
        };
        h->big_clusters[0] = sms;
        h->big_clusters[1] = query((const void*)k_tc_gemm_big<G_DOWN, 2>, 2, 1024 + big_smem_bytes<2>());
        h->big_clusters[2] = query((const void*)k_tc_gemm_big<G_DOWN, 4>, 4, 1024 + big_smem_bytes<4>());
        h->big_clusters[3] = query((const void*)k_tc_gemm_big<G_DOWN, 8>, 8, 1024 + big_smem_bytes<8>());
    }
    // JPI_BIG_SPLIT=S fixes the K split of the large-M residual projections (1, 2, 4 or 8).
    const char* split_env = std::getenv("JPI_BIG_SPLIT");
    if (split_env) h->big_split = std::atoi(split_env);
    // Launches with at least this many tokens use the large-M kernels (full K per CTA). The
    // gate/up projection (64 weight tiles at pi0.5 sizes) fills the GPU with them from 128 tokens;
    // the narrower ones (8-20 weight tiles) keep the K-split kernel up to 512 tokens (measured).
    // JPI_BIG_GEMM_MIN_TOKENS sets one threshold for all four.
    const char* big_env = std::getenv("JPI_BIG_GEMM_MIN_TOKENS");
    if (big_env)
        for (int k = 0; k < 4; ++k) h->big_min_tokens[k] = std::atoi(big_env);
    const int rows[4] = {h->QKV, h->W, 2 * h->F, h->W};
    const int ks[4] = {h->W, h->HD, h->W, h->F};
    // The K split (and so the summation order) is chosen once per projection, for every batch
    // size: a request's result does not depend on how many other requests share its batch.
    for (int g = 0; g < 4; ++g) {
        if (!make_plan(rows[g], ks[g], max_cluster, sms, g == G_QKV || g == G_GU, &h->plans[g])) {
            set_error("no tensor-core tiling for a %d x %d projection", rows[g], ks[g]);
            return JPI_ERR_UNSUPPORTED;
        }
    }
    // A cluster of `splits` CTAs must fit on the device at this shared-memory size.
    for (int g = 0; g < 4; ++g) {
        const GemmPlan& pl = h->plans[g];
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(pl.ctas);
        cfg.blockDim = dim3(GEMM_THREADS);
        cfg.dynamicSmemBytes = pl.smem;
        cudaLaunchAttribute at;
        at.id = cudaLaunchAttributeClusterDimension;
        at.val.clusterDim.x = pl.splits;
        at.val.clusterDim.y = 1;
        at.val.clusterDim.z = 1;
        cfg.attrs = &at;
        cfg.numAttrs = 1;
        int nclusters = 0;
        const void* fn = g == 0 ? (const void*)k_tc_gemm<G_QKV>
                       : g == 1 ? (const void*)k_tc_gemm<G_O>
                       : g == 2 ? (const void*)k_tc_gemm<G_GU>
                                : (const void*)k_tc_gemm<G_DOWN>;
        if (cudaOccupancyMaxActiveClusters(&nclusters, fn, &cfg) != cudaSuccess || nclusters < 1) {
            cudaGetLastError();
            set_error("a cluster of %d CTAs with %zu bytes of shared memory does not fit", pl.splits, pl.smem);
            return JPI_ERR_UNSUPPORTED;
        }
    }
    h->tmaps.resize((size_t)4 * h->L);
    for (int l = 0; l < h->L; ++l) {
        const LayerTiled& t = h->tiled[l];
        const int qkv_rows = h->QKV, o_rows = h->W, gu_rows = 2 * h->F, d_rows = h->W;
        JPI_TRY(make_tmap(t.qkv, (uint64_t)qkv_rows / TILE_ROWS * (h->W / KBLK) * TILE_ROWS, KBLK, TILE_ROWS,
                          &h->tmaps[4 * l + G_QKV]));
        JPI_TRY(make_tmap(t.o, (uint64_t)o_rows / TILE_ROWS * (h->HD / KBLK) * TILE_ROWS, KBLK, TILE_ROWS,
                          &h->tmaps[4 * l + G_O]));
        JPI_TRY(make_tmap(t.gu, (uint64_t)gu_rows / TILE_ROWS * (h->W / KBLK) * TILE_ROWS, KBLK, TILE_ROWS,
                          &h->tmaps[4 * l + G_GU]));
        JPI_TRY(make_tmap(t.down, (uint64_t)d_rows / TILE_ROWS * (h->F / KBLK) * TILE_ROWS, KBLK, TILE_ROWS,
                          &h->tmaps[4 * l + G_DOWN]));
    }
    // B operands: scaled residual stream in tiles of 63 tokens + beta, attention output and GeGLU
    // output ([rows][K] row-major).
    JPI_TRY(make_tmap(h->hx, (uint64_t)xs_tiles(h->maxMt) * 64, h->W, NT, &h->xmaps[0]));
    JPI_TRY(make_tmap(h->o, h->maxMt, h->HD, NT, &h->xmaps[1]));
    JPI_TRY(make_tmap(h->z, h->maxMt, h->F, NT, &h->xmaps[2]));
    JPI_TRY(mod_tc_prepare(h));
    // JPI_BATCH_INVARIANT=1: every launch makes the choices it makes for one request (K-split
    // projections, split-KV attention with a single request's key split), so a request's result
    // is the same bit for bit alone and inside any batch, at the cost of the batched kernels.
    const char* inv_env = std::getenv("JPI_BATCH_INVARIANT");
    if (inv_env && inv_env[0] == '1') {
        h->batch_invariant = true;
        h->attn_t5_min_batch = 0;
        for (int k = 0; k < 4; ++k) h->big_min_tokens[k] = 0;
    }
    return JPI_OK;
}

jpi_status tc_launch_op(jpi_handle* h, int op, int l, int step, int B, int C, cudaStream_t st) {
    const int W = h->W;
    const float* ms = h->mods + (size_t)step * mod_rows(h->L) * W + (size_t)6 * l * W;
    const size_t kv_layer = (size_t)l * h->maxB * h->kv_rows * h->D;
    const jpi::GemmPlan* plans = h->plans;
    const int Mt = B * (C + h->n_ctx());
    // Batched launches with many tokens: one CTA per (weight tile, 128-row operand tile) over
    // the whole K range. Residual kinds then leave one sum-of-squares slot per weight tile, and
    // the norm-fed kind after them reads as many slots as its producer left.
    auto big = [&](int kind) { return h->big_min_tokens[kind] > 0 && Mt >= h->big_min_tokens[kind]; };
    auto slots_left = [&](int kind) { return big(kind) ? plans[kind].ntiles : plans[kind].ntiles * plans[kind].splits; };
    auto run = [&](auto kind_tag, const GemmPlan& pl, const CUtensorMap& wm, const CUtensorMap& xm,
                   const GemmArgs& a) -> jpi_status {
        constexpr int KIND = decltype(kind_tag)::value;
        return big(KIND) ? launch_gemm_big<KIND>(h, pl, wm, xm, a, st) : launch_gemm<KIND>(h, pl, wm, xm, a, st);
    };
    using KQ = std::integral_constant<int, G_QKV>;
    using KO = std::integral_constant<int, G_O>;
    using KG = std::integral_constant<int, G_GU>;
    using KD = std::integral_constant<int, G_DOWN>;
    switch (op) {
        case 2: {
            const GemmPlan& pl = plans[G_QKV];
            GemmArgs a = base_args(h, B, C, pl);
            // Sums of squares left by the embedding (one per 128 features) or the previous
            // layer's down projection (one per CTA).
            if (l > 0) a.nslot = slots_left(G_DOWN);
            a.q = (__nv_bfloat16*)h->q;
            a.kst = (__nv_bfloat16*)h->kv_k + kv_layer;
            a.vst = (__nv_bfloat16*)h->kv_v + kv_layer;
            a.rope = h->rope_tab;
            return run(KQ{}, pl, h->tmaps[4 * l + G_QKV], h->xmaps[0], a);
        }
        case 3:
            // Batched launches: one CTA per 128 query rows over all keys (tcgen05, no split);
            // otherwise the split-KV kernel that spreads one request over the whole GPU.
            if (h->attn_t5 && h->attn_t5_min_batch > 0 && B >= h->attn_t5_min_batch)
                return launch_attn_t5(h, l, B, C, st);
            return attn_tc_supported(h) ? launch_attn_tc(h, l, B, C, st)
                                        : launch_op_simt(h, 3, l, step, B, C, st);
        case 4: {
            const GemmPlan& pl = plans[G_O];
            GemmArgs a = base_args(h, B, C, pl);
            a.hres = h->h;
            a.xs = (__nv_bfloat16*)h->hx;
            a.sigma_next = ms + 3 * W;   // the MLP norm of this layer
            a.beta_next = ms + 4 * W;
            a.gamma = ms + 2 * W;
            a.ss_out = h->ss;
            return run(KO{}, pl, h->tmaps[4 * l + G_O], h->xmaps[1], a);
        }
        case 5: {
            const GemmPlan& pl = plans[G_GU];
            GemmArgs a = base_args(h, B, C, pl);
            a.nslot = slots_left(G_O);   // left by O
            a.z = (__nv_bfloat16*)h->z;
            return run(KG{}, pl, h->tmaps[4 * l + G_GU], h->xmaps[0], a);
        }
        case 6: {
            const GemmPlan& pl = plans[G_DOWN];
            GemmArgs a = base_args(h, B, C, pl);
            a.hres = h->h;
            if (l + 1 < h->L) {           // the attention norm of the next layer
                a.xs = (__nv_bfloat16*)h->hx;
                a.sigma_next = ms + 6 * W;
                a.beta_next = ms + 7 * W;
            }
            a.gamma = ms + 5 * W;
            a.ss_out = h->ss;
            return run(KD{}, pl, h->tmaps[4 * l + G_DOWN], h->xmaps[2], a);
        }
        default:
            set_error("unknown layer op %d", op);
            return JPI_ERR_INVALID_ARG;
    }
}

jpi_status tc_launch_layer(jpi_handle* h, int l, int step, int B, int C, cudaStream_t st) {
    for (int op = 2; op <= 6; ++op) JPI_TRY(tc_launch_op(h, op, l, step, B, C, st));
    return JPI_OK;
}

void tc_release(jpi_handle*) {}

}  // namespace jpi
