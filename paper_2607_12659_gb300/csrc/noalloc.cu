// jpi_expert_forward_noalloc: one expert evaluation whose time-conditioning scratch lives in a
// fixed device array compiled into the library (see include/jpi.h for the contract).

#include "jpi_internal.h"
#include "tc_path.h"

#include <cstdio>

namespace {

// Largest width and time-embedding size the fixed scratch serves.
constexpr int NOALLOC_MAX_DIM = 8192;

// Scratch of the time-conditioning stage: sinusoidal embedding [d_t], time-MLP hidden layer
// [W] and conditioning vector [W]. Every GPU that loads the library holds these 96 KiB until
// the process exits. All three are overwritten in full by every call, so nothing needs
// clearing; calls that overlap on the GPU share them and race.
static __device__ __align__(256) float g_noalloc_tc_scratch[3 * NOALLOC_MAX_DIM];

// Device address of the array, resolved once per device (host code may not use the symbol
// itself: on the host it names a stand-in, not device memory).
constexpr int MAX_DEVICES = 64;
float* g_scratch_addr[MAX_DEVICES] = {};

jpi_status fail(jpi_status s, const char* msg) {
    jpi::set_error("%s", msg);
    return s;
}

}  // namespace

extern "C" JPI_API jpi_status jpi_expert_forward_noalloc(jpi_handle* h, const float* state,
                                                         const float* x_t, float t, int batch,
                                                         int chunk, float* out_v, float* out_h,
                                                         void* stream) {
    jpi::clear_error();
    if (!h) return fail(JPI_ERR_INVALID_ARG, "handle is NULL");
    if (!state || !x_t || !out_v) return fail(JPI_ERR_INVALID_ARG, "NULL input or output");
    if (batch < 1 || chunk < 1) return fail(JPI_ERR_INVALID_ARG, "batch and chunk must be >= 1");
    if (!(t >= 0.f)) return fail(JPI_ERR_INVALID_ARG, "t must be >= 0");
    if (batch > h->maxB || chunk > h->maxC) return fail(JPI_ERR_SHAPE, "batch or chunk exceeds the handle's maxima");
    if (!h->prefix_ready) return fail(JPI_ERR_NOT_READY, "no prefix KV has been set");
    if (batch != h->cur_batch) return fail(JPI_ERR_SHAPE, "batch differs from the prefix KV's batch");
    if (h->W > NOALLOC_MAX_DIM || h->dt > NOALLOC_MAX_DIM)
        return fail(JPI_ERR_SHAPE, "width or time_dim exceeds the fixed scratch (8192)");

    int dev = 0;
    JPI_CUDA_TRY(cudaGetDevice(&dev));
    if (dev < 0 || dev >= MAX_DEVICES) return fail(JPI_ERR_UNSUPPORTED, "device ordinal above 63");
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        JPI_CUDA_TRY(cudaGetSymbolAddress(&p, g_noalloc_tc_scratch));
        g_scratch_addr[dev] = (float*)p;
    }
    float* temb = g_scratch_addr[dev];
    float* c1 = temb + NOALLOC_MAX_DIM;
    float* cond = c1 + NOALLOC_MAX_DIM;

    cudaStream_t st = (cudaStream_t)stream;
    JPI_CUDA_TRY(cudaMemcpyAsync(h->state, state, (size_t)batch * h->Sd * sizeof(float),
                                 cudaMemcpyDeviceToDevice, st));
    JPI_CUDA_TRY(cudaMemcpyAsync(h->x, x_t, (size_t)batch * chunk * h->A * sizeof(float),
                                 cudaMemcpyDeviceToDevice, st));
    JPI_TRY(jpi::launch_time_conditioning_into(h, (double)t, temb, c1, cond, st));
    JPI_TRY(jpi::launch_embed(h, 0, batch, chunk, h->x, st));
    for (int l = 0; l < h->L; ++l) {
        if (h->tc)
            JPI_TRY(jpi::tc_launch_layer(h, l, 0, batch, chunk, st));
        else
            JPI_TRY(jpi::launch_layer_simt(h, l, 0, batch, chunk, st));
    }
    JPI_TRY(jpi::launch_final(h, 0, batch, chunk, 0.f, nullptr, out_v, nullptr, st));
    if (out_h)
        JPI_CUDA_TRY(cudaMemcpyAsync(out_h, h->h, (size_t)batch * (chunk + h->n_ctx()) * h->W * sizeof(float),
                                     cudaMemcpyDeviceToDevice, st));
    return JPI_OK;
}
