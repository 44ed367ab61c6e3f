// Launchers of the tcgen05 attention kernel (attn_t5_kernel.cuh) for the expert's batched
// denoise: one CTA per 128 query rows of a request and key split. The keys are split four ways
// when the (row blocks x requests) clusters of 4 CTAs are co-resident, else two ways when clusters
// of 2 are, else not at all (pi0.5 shapes, 4 row blocks per request: 4 at 3-9 requests, 2 at
// 10-19, 1 from 20).

#include "jpi_internal.h"
#include "ptx.h"
#include "tc_path.h"
#include "attn_t5_kernel.cuh"

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstdlib>

namespace jpi {
namespace {

static_assert(T5_ERR_LOAD == DEV_TIMEOUT_WEIGHTS && T5_ERR_MMA == DEV_TIMEOUT_MMA,
              "the attention kernel reports the library's device error codes");

constexpr int T5_MAX_SPLIT = 4;

// Whether `blocks` clusters of s CTAs are co-resident (one wave) and fit the workspace.
bool t5_fits(const jpi_handle* h, int blocks, int s) {
    return (long long)blocks * s <= h->num_sms && blocks <= h->t5_clusters[s];
}

int t5_splits(const jpi_handle* h, int blocks, int nb_all) {
    if (h->attn_t5_splits > 0) {
        // A fixed split, within the key blocks and one wave of clusters.
        int s = std::max(1, std::min({h->attn_t5_splits, T5_MAX_SPLIT, nb_all}));
        while (s > 1 && !t5_fits(h, blocks, s)) --s;
        return s;
    }
    // Four splits, else two, where the clusters fit in one wave; else none. A cluster past one
    // wave makes the launch take twice as long, and three splits pack fewer clusters than two or
    // four and keep no rows on chip.
    for (int s = T5_MAX_SPLIT; s >= 2; s /= 2)
        if (nb_all >= s && t5_fits(h, blocks, s)) return s;
    return 1;
}

template <int D>
jpi_status prepare_t5(jpi_handle* h) {
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_attn_t5<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      1024 + T5Smem<D>::TOTAL));
    // Co-resident clusters of s CTAs along z (the key splits of one row block).
    h->t5_clusters[1] = h->num_sms;
    for (int s = 2; s <= T5_MAX_SPLIT; ++s) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)(h->num_sms / s), 1, (unsigned)s);
        cfg.blockDim = dim3(T5_THREADS);
        cfg.dynamicSmemBytes = 1024 + T5Smem<D>::TOTAL;
        cudaLaunchAttribute at;
        at.id = cudaLaunchAttributeClusterDimension;
        at.val.clusterDim.x = 1;
        at.val.clusterDim.y = 1;
        at.val.clusterDim.z = (unsigned)s;
        cfg.attrs = &at;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, k_attn_t5<D>, &cfg) != cudaSuccess) {
            cudaGetLastError();
            n = 0;
        }
        h->t5_clusters[s] = n;
    }
    return JPI_OK;
}

template <int D>
jpi_status launch_t5(jpi_handle* h, int l, int B, int C, cudaStream_t st) {
    T5Args a;
    a.S = C + h->n_ctx();
    a.nctx = h->n_ctx();
    a.H = h->H;
    a.P = h->cur_prefix;
    a.kv_rows = h->kv_rows;
    a.maxB = h->maxB;
    a.layer = l;
    const int rblocks = (a.S * a.H + T5_ROWS - 1) / T5_ROWS;
    a.scale_log2 = 1.4426950408889634f / sqrtf((float)D);
    a.o = (__nv_bfloat16*)h->o;
    a.err = h->dev_err;
    const int splits = h->t5_ws ? t5_splits(h, rblocks * B, (a.P + a.S + T5_KEYS - 1) / T5_KEYS) : 1;
    a.ws = reinterpret_cast<float4*>(h->t5_ws);
    a.wml = reinterpret_cast<float2*>(h->t5_wml);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(rblocks, B, splits);
    cfg.blockDim = dim3(T5_THREADS);
    cfg.dynamicSmemBytes = 1024 + T5Smem<D>::TOTAL;
    cfg.stream = st;
    cudaLaunchAttribute attrs[2];
    int n = 0;
    if (h->pdl) {
        attrs[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attrs[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    if (splits > 1) {
        attrs[n].id = cudaLaunchAttributeClusterDimension;
        attrs[n].val.clusterDim.x = 1;
        attrs[n].val.clusterDim.y = 1;
        attrs[n].val.clusterDim.z = (unsigned)splits;
        ++n;
    }
    cfg.attrs = attrs;
    cfg.numAttrs = n;
    cudaError_t e = cudaLaunchKernelEx(&cfg, k_attn_t5<D>, h->amaps[0], h->amaps[1], h->amaps[2], a);
    if (e != cudaSuccess) {
        set_error("attention launch failed: %s", cudaGetErrorString(e));
        return JPI_ERR_CUDA;
    }
    return JPI_OK;
}

}  // namespace

bool attn_t5_supported(const jpi_handle* h) {
    return h->bf16 && (h->D == 128 || h->D == 256);
}

jpi_status attn_t5_prepare(jpi_handle* h) {
    if (!attn_t5_supported(h)) return JPI_OK;
    // Smallest batch that takes this kernel (smaller ones keep the split-KV kernel); the
    // environment can move it, 0 turns the kernel off.
    const char* env = std::getenv("JPI_ATTN_T5_MIN_BATCH");
    h->attn_t5_min_batch = env ? std::atoi(env) : 3;
    // JPI_ATTN_T5_SPLITS fixes its key split (1, 2 or 4; 0 or unset: chosen per launch).
    const char* split_env = std::getenv("JPI_ATTN_T5_SPLITS");
    h->attn_t5_splits = split_env ? std::atoi(split_env) : 0;
    // Workspace of the key splits: a slot per CTA of a launch that splits (at most one CTA per SM).
    {
        const size_t part = (size_t)h->num_sms * (h->D / 4) * T5_ROWS * sizeof(float4);
        const size_t ml = (size_t)h->num_sms * T5_ROWS * sizeof(float2);
        void* p = nullptr;
        if (cudaMalloc(&p, part + ml) != cudaSuccess) {
            cudaGetLastError();
            set_error("cudaMalloc of %zu bytes failed", part + ml);
            return JPI_ERR_OOM;
        }
        h->allocations.push_back(p);
        h->device_bytes += part + ml;
        h->t5_ws = p;
        h->t5_wml = static_cast<uint8_t*>(p) + part;
    }
    // q [maxMt * H][D]; K and V of all layers [L * maxB * kv_rows][D].
    JPI_TRY(tc_make_tmap(h->q, (uint64_t)h->maxMt * h->H, h->D, T5_ROWS, &h->amaps[0]));
    const uint64_t kv_rows_all = (uint64_t)h->L * h->maxB * h->kv_rows;
    JPI_TRY(tc_make_tmap(h->kv_k, kv_rows_all, h->D, T5_KEYS, &h->amaps[1]));
    JPI_TRY(tc_make_tmap(h->kv_v, kv_rows_all, h->D, T5_KEYS, &h->amaps[2]));
    JPI_TRY(h->D == 256 ? prepare_t5<256>(h) : prepare_t5<128>(h));
    h->attn_t5 = true;
    return JPI_OK;
}

jpi_status launch_attn_t5(jpi_handle* h, int l, int B, int C, cudaStream_t st) {
    return h->D == 256 ? launch_t5<256>(h, l, B, C, st) : launch_t5<128>(h, l, B, C, st);
}

}  // namespace jpi
