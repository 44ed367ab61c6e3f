// Tensor-core path of the bf16 expert layers: tcgen05 GEMMs fed by bulk tensor copies.
//
// Every projection of a layer is a skinny GEMM Y[tokens][out] = X[tokens][K] W[out][K]^T with
// tokens = batch x (chunk + 1) (51 at batch 1). It runs "swap-AB": a 128-row tile of W is the
// A operand (M = 128), a 64-token tile of X is the B operand (N = 64), and the fp32 product
// sits in TMEM. The K dimension of each weight tile is split across the CTAs of one thread-
// block cluster; each CTA loads its weight blocks with bulk tensor copies before it waits on
// the previous kernel (weights do not depend on it), then builds its X blocks in shared
// memory with the previous op's normalisation fused in, multiplies, and the cluster reduces
// its fp32 partials through distributed shared memory in a fixed rank order, so results do
// not depend on timing. Each CTA applies the epilogue to its slice of the reduced tile:
// rotary encoding + scatter into the query buffer and KV store (QKV), GeGLU (gate/up), or the
// gated residual update with per-token sums of squares for the next RMSNorm (O, down).

#include "tc_path.h"
#include "ptx.h"

#include <cooperative_groups.h>
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <vector>

namespace cg = cooperative_groups;

namespace jpi {
namespace {

constexpr int NT = 64;                         // tokens per MMA (N)
constexpr int TILE_ROWS = 128;                 // weight rows per tile (M)
constexpr int KBLK = 64;                       // K elements per block: one 128-byte swizzle row
constexpr int TILE_BYTES = TILE_ROWS * KBLK * 2;
constexpr int XBLK_BYTES = NT * KBLK * 2;
constexpr int PSTRIDE = NT + 4;                // fp32 partial row stride (floats)
constexpr int GEMM_THREADS = 128;
constexpr int MAX_SPLITS = 16;
constexpr uint64_t WAIT_LIMIT_NS = 200ull * 1000 * 1000;   // 0.2 s

enum GemmKind { G_QKV = 0, G_O = 1, G_GU = 2, G_DOWN = 3 };

struct GemmArgs {
    int Mt, K, nkb, kpb, splits;
    // RMSNorm-modulated input (QKV, gate/up): u = h * rinv * (1 + sigma) + beta.
    const float* h;
    const float* ss;         // [nslot][ss_ld] per-token sums of squares of h over 128 features
    int nslot, ss_ld;
    const float* sigma;
    const float* beta;
    float eps, inv_w;
    // bf16 input (O-proj, down).
    const __nv_bfloat16* act;
    // Gated residual epilogue.
    float* hres;
    const float* gamma;
    float* ss_out;
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

__device__ __forceinline__ float gelu_tanh(float y) {
    const float k0 = 0.7978845608028654f;   // sqrt(2 / pi)
    return 0.5f * y * (1.f + tanhf(k0 * (y + 0.044715f * y * y * y)));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ void set_device_error(int* err, int code) { atomicCAS(err, 0, code); }

template <int KIND>
__device__ __forceinline__ void epilogue(const GemmArgs& a, int tile, int p, int tok, float y1,
                                         float y2, float& ssacc) {
    if (KIND == G_QKV) {
        const int hd = a.D >> 1;
        const int pair = tile * 64 + p;
        const int sec = pair / hd, d = pair - sec * hd;     // sec < H: query head, H: key, H+1: value
        const int b = tok / a.S, i = tok - b * a.S, pos = a.P + i;
        if (sec <= a.H) {
            float c = 1.f, s = 0.f;
            if (a.rope) {
                const float2 cs = a.rope[(size_t)pos * hd + d];
                c = cs.x;
                s = cs.y;
            }
            const float r1 = y1 * c - y2 * s, r2 = y2 * c + y1 * s;
            __nv_bfloat16* dst = (sec < a.H) ? a.q + ((size_t)tok * a.H + sec) * a.D
                                             : a.kst + ((size_t)b * a.kv_rows + pos) * a.D;
            dst[d] = __float2bfloat16_rn(r1);
            dst[d + hd] = __float2bfloat16_rn(r2);
        } else {
            __nv_bfloat16* dst = a.vst + ((size_t)b * a.kv_rows + pos) * a.D;
            dst[d] = __float2bfloat16_rn(y1);
            dst[d + hd] = __float2bfloat16_rn(y2);
        }
    } else if (KIND == G_GU) {
        const int f = tile * 64 + p;
        a.z[(size_t)tok * a.F + f] = __float2bfloat16_rn(gelu_tanh(y1) * y2);
    } else {
        const int f1 = tile * TILE_ROWS + p, f2 = f1 + 64;
        float* hr = a.hres + (size_t)tok * a.W;
        const float n1 = hr[f1] + a.gamma[f1] * y1;
        const float n2 = hr[f2] + a.gamma[f2] * y2;
        hr[f1] = n1;
        hr[f2] = n2;
        ssacc = fmaf(n1, n1, ssacc);
        ssacc = fmaf(n2, n2, ssacc);
    }
}

template <int KIND>
__global__ void __launch_bounds__(GEMM_THREADS) k_tc_gemm(const __grid_constant__ CUtensorMap tmap,
                                                          const __grid_constant__ GemmArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const int xp_bytes = max(a.kpb * XBLK_BYTES, TILE_ROWS * PSTRIDE * 4);
    uint8_t* wsm = smem;                                   // kpb weight tiles
    uint8_t* xsm = wsm + a.kpb * TILE_BYTES;               // X blocks, then the fp32 partial
    float* part = (float*)xsm;
    float* slots = (float*)(xsm + xp_bytes);               // [MAX_SPLITS][NT] (rank 0)
    float* rinv = slots + MAX_SPLITS * NT;                 // [NT]
    float* sspair = rinv + NT;                             // [GEMM_THREADS]
    uint64_t* bars = (uint64_t*)(sspair + GEMM_THREADS);   // [0] weights, [1] MMA done
    uint32_t* tmem_slot = (uint32_t*)(bars + 2);
    int* flag = (int*)(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int tile = blockIdx.x / a.splits;
    const int kb0 = rank * a.kpb;

    if (warp == 0) {
        ptx::tmem_alloc(tmem_slot, NT);
        ptx::tmem_relinquish();
    }
    if (tid == 0) {
        ptx::mbar_init(&bars[0], 1);
        ptx::mbar_init(&bars[1], 1);
        ptx::fence_mbar_init();
        *flag = 0;
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    // Weight tiles depend on nothing upstream: start streaming them before the dependency wait.
    if (tid == 0) {
        const uint64_t pol = ptx::l2_policy_evict_first();
        ptx::mbar_expect_tx(&bars[0], (uint32_t)(a.kpb * TILE_BYTES));
        for (int j = 0; j < a.kpb; ++j)
            ptx::tma_load_2d(wsm + j * TILE_BYTES, &tmap, &bars[0], 0,
                             (tile * a.nkb + kb0 + j) * TILE_ROWS, pol);
    }
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();

    const int ntt = (a.Mt + NT - 1) / NT;
    const int npairs = 64 / a.splits, p0 = rank * npairs;
    constexpr bool NORM_IN = (KIND == G_QKV || KIND == G_GU);
    constexpr bool RESID = (KIND == G_O || KIND == G_DOWN);
    constexpr uint32_t IDESC = ptx::idesc_bf16_f32(TILE_ROWS, NT);

    for (int tt = 0; tt < ntt; ++tt) {
        const int tok0 = tt * NT;
        // ---- B operand: X[tok][kb0*64 .. (kb0+kpb)*64) in the 128-byte swizzle layout ----
        if (NORM_IN) {
            if (tid < NT) {
                const int tok = tok0 + tid;
                float r = 0.f;
                if (tok < a.Mt) {
                    float s = 0.f;
                    for (int sl = 0; sl < a.nslot; ++sl) s += a.ss[(size_t)sl * a.ss_ld + tok];
                    r = rsqrtf(s * a.inv_w + a.eps);
                }
                rinv[tid] = r;
            }
            __syncthreads();
        }
        for (int idx = tid; idx < a.kpb * NT * 8; idx += GEMM_THREADS) {
            const int j = idx / (NT * 8), t = (idx >> 3) % NT, c = idx & 7;
            const int tok = tok0 + t, k = (kb0 + j) * KBLK + c * 8;
            uint4 v = make_uint4(0u, 0u, 0u, 0u);
            if (tok < a.Mt) {
                if (NORM_IN) {
                    const float4* hp = (const float4*)(a.h + (size_t)tok * a.K + k);
                    const float4* sp = (const float4*)(a.sigma + k);
                    const float4* bp = (const float4*)(a.beta + k);
                    const float r = rinv[t];
                    const float4 h0 = hp[0], h1 = hp[1], s0 = sp[0], s1 = sp[1], b0 = bp[0], b1 = bp[1];
                    v.x = pack_bf16x2(h0.x * r * (1.f + s0.x) + b0.x, h0.y * r * (1.f + s0.y) + b0.y);
                    v.y = pack_bf16x2(h0.z * r * (1.f + s0.z) + b0.z, h0.w * r * (1.f + s0.w) + b0.w);
                    v.z = pack_bf16x2(h1.x * r * (1.f + s1.x) + b1.x, h1.y * r * (1.f + s1.y) + b1.y);
                    v.w = pack_bf16x2(h1.z * r * (1.f + s1.z) + b1.z, h1.w * r * (1.f + s1.w) + b1.w);
                } else {
                    v = *(const uint4*)(a.act + (size_t)tok * a.K + k);
                }
            }
            *(uint4*)(xsm + j * XBLK_BYTES + t * 128 + ((c ^ (t & 7)) << 4)) = v;
        }
        ptx::fence_proxy_async_smem();
        __syncthreads();

        // ---- MMA: D[128 rows][NT tokens] = sum over this CTA's K blocks ----
        if (tid == 0 && *flag == 0) {
            if (tt == 0 && !ptx::mbar_wait_bounded(&bars[0], 0, WAIT_LIMIT_NS)) {
                *flag = DEV_TIMEOUT_WEIGHTS;
            } else {
                ptx::tc_fence_after();
                const uint32_t wbase = ptx::smem_u32(wsm), xbase = ptx::smem_u32(xsm);
                for (int j = 0; j < a.kpb; ++j)
#pragma unroll
                    for (int kk = 0; kk < KBLK / 16; ++kk)
                        ptx::mma_bf16(tmem, ptx::desc_sw128(wbase + j * TILE_BYTES + kk * 32),
                                      ptx::desc_sw128(xbase + j * XBLK_BYTES + kk * 32), IDESC,
                                      (j | kk) != 0);
                ptx::mma_commit(&bars[1]);
            }
        }
        __syncthreads();
        if (*flag == 0 && !ptx::mbar_wait_bounded(&bars[1], tt & 1, WAIT_LIMIT_NS)) *flag = DEV_TIMEOUT_MMA;
        __syncthreads();
        const bool ok = *flag == 0;
        ptx::tc_fence_after();

        // ---- TMEM -> fp32 partial in shared memory (thread = row) ----
        if (ok) {
            const int row = warp * 32 + lane;
#pragma unroll
            for (int c0 = 0; c0 < NT; c0 += 16) {
                uint32_t r[16];
                ptx::tmem_ld_x16(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)c0, r);
                ptx::tmem_ld_wait();
                float4* dst = (float4*)(part + row * PSTRIDE + c0);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4)
                    dst[q4] = make_float4(__uint_as_float(r[4 * q4]), __uint_as_float(r[4 * q4 + 1]),
                                          __uint_as_float(r[4 * q4 + 2]), __uint_as_float(r[4 * q4 + 3]));
            }
        }
        ptx::tc_fence_before();
        cluster.sync();

        // ---- cluster reduction in rank order + epilogue on this CTA's row pairs ----
        float ssacc = 0.f;
        for (int idx = tid; idx < npairs * NT; idx += GEMM_THREADS) {
            const int p = p0 + idx / NT, t = idx % NT, tok = tok0 + t;
            float y1 = 0.f, y2 = 0.f;
            for (int r = 0; r < a.splits; ++r) {
                const float* rp = cluster.map_shared_rank(part, r);
                y1 += rp[p * PSTRIDE + t];
                y2 += rp[(p + 64) * PSTRIDE + t];
            }
            if (tok < a.Mt && ok) epilogue<KIND>(a, tile, p, tok, y1, y2, ssacc);
        }
        if (RESID) {
            sspair[tid] = ssacc;
            __syncthreads();
            if (tid < NT) {
                float s = 0.f;
                for (int q = tid; q < GEMM_THREADS; q += NT) s += sspair[q];
                float* rs = cluster.map_shared_rank(slots, 0);
                rs[rank * NT + tid] = s;
            }
        }
        cluster.sync();
        if (RESID && rank == 0 && tid < NT && ok) {
            const int tok = tok0 + tid;
            if (tok < a.Mt) {
                float s = 0.f;
                for (int r = 0; r < a.splits; ++r) s += slots[r * NT + tid];
                a.ss_out[(size_t)tile * a.ss_ld + tok] = s;
            }
        }
    }

    if (tid == 0 && *flag != 0) set_device_error(a.err, *flag);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 0) ptx::tmem_dealloc(tmem, NT);
}

// ---------------------------------------------------------------------------------------------
// Host side: packing, plans, tensor maps, launches.

size_t gemm_smem(int kpb) {
    const size_t xp = std::max((size_t)kpb * XBLK_BYTES, (size_t)TILE_ROWS * PSTRIDE * 4);
    return 1024 + (size_t)kpb * TILE_BYTES + xp + sizeof(float) * (MAX_SPLITS * NT + NT + GEMM_THREADS) + 64;
}

bool make_plan(int rows, int K, int max_cluster, int num_sms, GemmPlan* out) {
    if (rows % TILE_ROWS || K % KBLK) return false;
    GemmPlan best;
    long best_score = -1;
    const int ntiles = rows / TILE_ROWS, nkb = K / KBLK;
    for (int kpb = 1; kpb <= 8; kpb *= 2) {
        if (nkb % kpb) continue;
        const int splits = nkb / kpb;
        if (splits > max_cluster || 64 % splits) continue;
        const size_t smem = gemm_smem(kpb);
        if (smem > 227 * 1024) continue;
        const int res = std::min(4, (int)((228 * 1024) / (smem + 1024)));
        const int ctas = ntiles * splits;
        const long waves = (ctas + (long)num_sms * res - 1) / ((long)num_sms * res);
        const long per_sm = (ctas + num_sms - 1) / num_sms;
        const long score = waves * 1000 + per_sm * kpb * 10 + (ctas > num_sms ? 1 : 0);
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

jpi_status make_tmap(const __nv_bfloat16* base, const GemmPlan& pl, CUtensorMap* map) {
    auto enc = get_encode();
    if (!enc) {
        set_error("cuTensorMapEncodeTiled is unavailable from the driver");
        return JPI_ERR_CUDA;
    }
    const cuuint64_t dims[2] = {(cuuint64_t)KBLK, (cuuint64_t)pl.ntiles * pl.nkb * TILE_ROWS};
    const cuuint64_t strides[1] = {(cuuint64_t)KBLK * 2};
    const cuuint32_t box[2] = {(cuuint32_t)KBLK, (cuuint32_t)TILE_ROWS};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void*)base, dims, strides, box, estr,
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
jpi_status launch_gemm(jpi_handle* h, const GemmPlan& pl, const CUtensorMap& map, const GemmArgs& a,
                       cudaStream_t st) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(pl.ctas);
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
    cudaError_t e = cudaLaunchKernelEx(&cfg, k_tc_gemm<KIND>, map, a);
    if (e != cudaSuccess) {
        set_error("tensor-core GEMM launch failed: %s", cudaGetErrorString(e));
        return JPI_ERR_CUDA;
    }
    return JPI_OK;
}

GemmArgs base_args(jpi_handle* h, int B, int C, const GemmPlan& pl) {
    GemmArgs a = {};
    a.Mt = B * (C + 1);
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
    a.S = C + 1;
    a.H = h->H;
    a.D = h->D;
    a.P = h->cur_prefix;
    a.kv_rows = h->kv_rows;
    a.F = h->F;
    a.err = h->dev_err;
    return a;
}

}  // namespace

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
    const char* pdl_env = std::getenv("JPI_PDL");
    h->pdl = !(pdl_env && pdl_env[0] == '0');

    int max_cluster = 16;
    auto kernels = {k_tc_gemm<G_QKV>, k_tc_gemm<G_O>, k_tc_gemm<G_GU>, k_tc_gemm<G_DOWN>};
    for (auto k : kernels) {
        if (cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
            cudaGetLastError();
            max_cluster = 8;
        }
        JPI_CUDA_TRY(cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)gemm_smem(8)));
    }
    const int rows[4] = {h->QKV, h->W, 2 * h->F, h->W};
    const int ks[4] = {h->W, h->HD, h->W, h->F};
    for (int g = 0; g < 4; ++g) {
        if (!make_plan(rows[g], ks[g], max_cluster, sms, &h->plans[g])) {
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
        JPI_TRY(make_tmap(t.qkv, h->plans[G_QKV], &h->tmaps[4 * l + G_QKV]));
        JPI_TRY(make_tmap(t.o, h->plans[G_O], &h->tmaps[4 * l + G_O]));
        JPI_TRY(make_tmap(t.gu, h->plans[G_GU], &h->tmaps[4 * l + G_GU]));
        JPI_TRY(make_tmap(t.down, h->plans[G_DOWN], &h->tmaps[4 * l + G_DOWN]));
    }
    return JPI_OK;
}

jpi_status tc_launch_op(jpi_handle* h, int op, int l, int step, int B, int C, cudaStream_t st) {
    const int W = h->W;
    const float* ms = h->mods + (size_t)step * mod_rows(h->L) * W + (size_t)6 * l * W;
    const size_t kv_layer = (size_t)l * h->maxB * h->kv_rows * h->D;
    switch (op) {
        case 2: {
            const GemmPlan& pl = h->plans[G_QKV];
            GemmArgs a = base_args(h, B, C, pl);
            a.h = h->h;
            a.sigma = ms;
            a.beta = ms + W;
            a.q = (__nv_bfloat16*)h->q;
            a.kst = (__nv_bfloat16*)h->kv_k + kv_layer;
            a.vst = (__nv_bfloat16*)h->kv_v + kv_layer;
            a.rope = h->rope_tab;
            return launch_gemm<G_QKV>(h, pl, h->tmaps[4 * l + G_QKV], a, st);
        }
        case 3:
            return launch_op_simt(h, 3, l, step, B, C, st);
        case 4: {
            const GemmPlan& pl = h->plans[G_O];
            GemmArgs a = base_args(h, B, C, pl);
            a.act = (const __nv_bfloat16*)h->o;
            a.hres = h->h;
            a.gamma = ms + 2 * W;
            a.ss_out = h->ss;
            return launch_gemm<G_O>(h, pl, h->tmaps[4 * l + G_O], a, st);
        }
        case 5: {
            const GemmPlan& pl = h->plans[G_GU];
            GemmArgs a = base_args(h, B, C, pl);
            a.h = h->h;
            a.sigma = ms + 3 * W;
            a.beta = ms + 4 * W;
            a.z = (__nv_bfloat16*)h->z;
            return launch_gemm<G_GU>(h, pl, h->tmaps[4 * l + G_GU], a, st);
        }
        case 6: {
            const GemmPlan& pl = h->plans[G_DOWN];
            GemmArgs a = base_args(h, B, C, pl);
            a.act = (const __nv_bfloat16*)h->z;
            a.hres = h->h;
            a.gamma = ms + 5 * W;
            a.ss_out = h->ss;
            return launch_gemm<G_DOWN>(h, pl, h->tmaps[4 * l + G_DOWN], a, st);
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
