// jpi_expert_forward_noalloc: one expert evaluation whose time-conditioning scratch lives in a
// fixed device array compiled into the library (see include/jpi.h for the contract).

#include "jpi_internal.h"
#include "tc_path.h"

#include <mutex>

namespace {

// Largest width and time-embedding size the fixed scratch serves.
constexpr int NOALLOC_MAX_DIM = 8192;

// Scratch of the time-conditioning stage: sinusoidal embedding [d_t], time-MLP hidden layer
// [W] and conditioning vector [W]. Every GPU that loads the library holds these 96 KiB until
// the process exits. All three are overwritten in full by every call, so nothing needs
// clearing; calls that overlap on the GPU share them and race.
static __device__ __align__(256) float g_noalloc_tc_scratch[3 * NOALLOC_MAX_DIM];

// Device address of the array per device, with the id of the CUDA context it was resolved in.
// Host code may not use the symbol itself: on the host it names a stand-in, not device memory.
// A new context on the device (after cudaDeviceReset, say) has a new id, and the address is
// resolved again.
constexpr int MAX_DEVICES = 64;
struct ScratchAddr {
    unsigned long long ctx_id = 0;
    bool valid = false;
    float* ptr = nullptr;
};
ScratchAddr g_scratch[MAX_DEVICES];
std::mutex g_scratch_mutex;

// Driver entry points for the current context's id, resolved through the runtime so that the
// library links no driver library.
typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

jpi_status current_context_id(unsigned long long* id) {
    static CtxGetCurrentFn get_current = nullptr;
    static CtxGetIdFn get_id = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess && q == cudaDriverEntryPointSuccess)
            get_current = (CtxGetCurrentFn)p;
        p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess && q == cudaDriverEntryPointSuccess)
            get_id = (CtxGetIdFn)p;
    });
    if (!get_current || !get_id) {
        jpi::set_error("cuCtxGetCurrent / cuCtxGetId are unavailable from the driver");
        return JPI_ERR_CUDA;
    }
    CUcontext ctx = nullptr;
    if (get_current(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, id) != CUDA_SUCCESS) {
        jpi::set_error("no current CUDA context on the calling thread");
        return JPI_ERR_CUDA;
    }
    return JPI_OK;
}

// The array's device address on `dev`, which is the calling thread's current device.
jpi_status scratch_address(int dev, float** out) {
    // Makes the device's primary context current on this thread if no call has done so yet.
    JPI_CUDA_TRY(cudaSetDevice(dev));
    unsigned long long id = 0;
    JPI_TRY(current_context_id(&id));
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    ScratchAddr& a = g_scratch[dev];
    if (!a.valid || a.ctx_id != id) {
        void* p = nullptr;
        JPI_CUDA_TRY(cudaGetSymbolAddress(&p, g_noalloc_tc_scratch));
        a.ptr = (float*)p;
        a.ctx_id = id;
        a.valid = true;
    }
    *out = a.ptr;
    return JPI_OK;
}

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
    JPI_TRY(jpi::check_call(h, batch, chunk, 1));
    if (!state || !x_t || !out_v) return fail(JPI_ERR_INVALID_ARG, "NULL input or output");
    if (!(t >= 0.f)) return fail(JPI_ERR_INVALID_ARG, "t must be >= 0");
    if (h->W > NOALLOC_MAX_DIM || h->dt > NOALLOC_MAX_DIM)
        return fail(JPI_ERR_SHAPE, "width or time_dim exceeds the fixed scratch (8192)");

    int dev = 0;
    JPI_CUDA_TRY(cudaGetDevice(&dev));
    if (dev != h->device)
        return fail(JPI_ERR_INVALID_ARG, "the calling thread's current device is not the handle's device");
    if (dev < 0 || dev >= MAX_DEVICES) return fail(JPI_ERR_UNSUPPORTED, "device ordinal above 63");
    float* temb = nullptr;
    JPI_TRY(scratch_address(dev, &temb));
    float* c1 = temb + NOALLOC_MAX_DIM;
    float* cond = c1 + NOALLOC_MAX_DIM;

    cudaStream_t st = (cudaStream_t)stream;
    JPI_CUDA_TRY(cudaMemcpyAsync(h->state, state, (size_t)batch * h->Sd * sizeof(float),
                                 cudaMemcpyDeviceToDevice, st));
    JPI_CUDA_TRY(cudaMemcpyAsync(h->x, x_t, (size_t)batch * chunk * h->A * sizeof(float),
                                 cudaMemcpyDeviceToDevice, st));
    JPI_TRY(jpi::launch_time_conditioning_into(h, (double)t, temb, c1, cond, st));
    JPI_TRY(jpi::enqueue_step(h, 0, batch, chunk, 0.f, out_v, st));
    if (out_h)
        JPI_CUDA_TRY(cudaMemcpyAsync(out_h, h->h, (size_t)batch * (chunk + h->n_ctx()) * h->W * sizeof(float),
                                     cudaMemcpyDeviceToDevice, st));
    return JPI_OK;
}
