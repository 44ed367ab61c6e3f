// Launchers of the tcgen05 attention kernel (attn_t5_kernel.cuh) for the expert's batched
// denoise: one CTA per 128 query rows of a request over its prefix and suffix keys, no key split.

#include "jpi_internal.h"
#include "ptx.h"
#include "tc_path.h"
#include "attn_t5_kernel.cuh"

#include <cmath>
#include <cstdlib>

namespace jpi {
namespace {

static_assert(T5_ERR_LOAD == DEV_TIMEOUT_WEIGHTS && T5_ERR_MMA == DEV_TIMEOUT_MMA,
              "the attention kernel reports the library's device error codes");

template <int D>
jpi_status prepare_t5(jpi_handle* h) {
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_attn_t5<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      1024 + T5Smem<D>::TOTAL));
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
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(rblocks, B);
    cfg.blockDim = dim3(T5_THREADS);
    cfg.dynamicSmemBytes = 1024 + T5Smem<D>::TOTAL;
    cfg.stream = st;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr.val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = h->pdl ? 1 : 0;
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
    h->attn_t5_min_batch = env ? std::atoi(env) : 6;
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
