// C-ABI entry points: argument checks, the handle's persistent buffers, weight packing, the
// GPU-resident prefix-KV store and the captured, unrolled N-step denoise graph.
//
// Sec. 4.3 of the paper ("System Design") motivates the runtime shape: the token length is
// fixed for a given prefix, so the denoise of one chunk is captured once as a CUDA graph with
// every Euler step unrolled into it and replayed afterwards; every intermediate lives in a
// fixed device buffer allocated once at create time.

#include "jpi_internal.h"
#include "tc_path.h"

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>

namespace jpi {

namespace {
thread_local char g_err[1024] = "";
}

void set_error(const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
}
void clear_error() { g_err[0] = '\0'; }

namespace {

jpi_status fail(jpi_status s, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return s;
}

template <typename T>
jpi_status dev_alloc(jpi_handle* h, T** p, size_t count) {
    void* q = nullptr;
    const size_t bytes = count * sizeof(T);
    cudaError_t e = cudaMalloc(&q, bytes ? bytes : 16);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(JPI_ERR_OOM, "cudaMalloc(%zu bytes) failed: %s", bytes, cudaGetErrorString(e));
    }
    h->allocations.push_back(q);
    h->device_bytes += bytes;
    *p = (T*)q;
    return JPI_OK;
}

// fp32 -> element type of the weight store (bf16 rounding to nearest, ties to even).
__global__ void k_f32_to_bf16(const float* __restrict__ src, __nv_bfloat16* __restrict__ dst,
                              long long n) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
         i += (long long)gridDim.x * blockDim.x)
        dst[i] = __float2bfloat16_rn(src[i]);
}

// Moves one fp32 source tensor (host or device) to `dst` as fp32 or bf16.
struct Uploader {
    jpi_handle* h;
    bool on_device;
    float* tmp = nullptr;       // device staging for host sources / conversion
    size_t tmp_elems = 0;

    jpi_status put(void* dst, bool to_bf16, const float* src, size_t n, const char* name) {
        if (!src) return fail(JPI_ERR_INVALID_ARG, "weight tensor %s is NULL", name);
        const float* dsrc = src;
        if (!on_device) {
            if (!to_bf16) {
                JPI_CUDA_TRY(cudaMemcpy(dst, src, n * sizeof(float), cudaMemcpyHostToDevice));
                return JPI_OK;
            }
            JPI_CUDA_TRY(cudaMemcpy(tmp, src, n * sizeof(float), cudaMemcpyHostToDevice));
            dsrc = tmp;
        }
        if (to_bf16) {
            const long long nn = (long long)n;
            int g = (int)((nn + 255) / 256);
            if (g > 8192) g = 8192;
            if (g < 1) g = 1;
            k_f32_to_bf16<<<g, 256>>>(dsrc, (__nv_bfloat16*)dst, nn);
            JPI_CUDA_TRY(cudaGetLastError());
        } else {
            JPI_CUDA_TRY(cudaMemcpy(dst, dsrc, n * sizeof(float), cudaMemcpyDeviceToDevice));
        }
        return JPI_OK;
    }
};

inline size_t tw_size(const jpi_handle* h) { return h->bf16 ? 2 : 4; }
inline void* tw_offset(const jpi_handle* h, void* base, size_t elems) {
    return (char*)base + elems * tw_size(h);
}

jpi_status check_config(const jpi_config* c) {
    if (!c) return fail(JPI_ERR_INVALID_ARG, "config is NULL");
    if (c->n_layers < 1 || c->width < 32 || c->width % 32 || c->n_heads < 1 || c->head_dim < 32 ||
        c->mlp_dim < 32 || c->action_dim < 1 || c->state_dim < 1 || c->time_dim < 4)
        return fail(JPI_ERR_INVALID_ARG, "config has a dimension below its minimum");
    if (c->n_kv_heads != 1) return fail(JPI_ERR_UNSUPPORTED, "n_kv_heads must be 1");
    if (c->time_dim % 2) return fail(JPI_ERR_INVALID_ARG, "time_dim must be even");
    if (c->head_dim % 32 || c->head_dim > 256)
        return fail(JPI_ERR_UNSUPPORTED, "head_dim must be a multiple of 32 and at most 256");
    if (c->n_heads > 32) return fail(JPI_ERR_UNSUPPORTED, "n_heads must be at most 32");
    if (c->max_batch < 1 || c->max_prefix < 1 || c->max_chunk < 1 || c->max_steps < 1)
        return fail(JPI_ERR_INVALID_ARG, "max_batch/max_prefix/max_chunk/max_steps must be >= 1");
    if (c->max_steps > 64) return fail(JPI_ERR_UNSUPPORTED, "max_steps must be at most 64");
    if (c->precision != JPI_BF16 && c->precision != JPI_FP32)
        return fail(JPI_ERR_INVALID_ARG, "unknown precision %d", (int)c->precision);
    if (!(c->rms_eps >= 0.f) || !(c->rope_base >= 0.f) || !(c->t_min_period > 0.f) ||
        !(c->t_max_period > 0.f))
        return fail(JPI_ERR_INVALID_ARG, "rms_eps/rope_base must be >= 0 and periods > 0");
    const long long mt = (long long)c->max_batch * (c->max_chunk + 1 + JPI_MAX_CORRECTION);
    if (mt > (1 << 20) || (long long)c->max_prefix > (1 << 20))
        return fail(JPI_ERR_SHAPE, "maxima too large");
    return JPI_OK;
}

jpi_status pack_weights(jpi_handle* h, const jpi_weights* w) {
    const int L = h->L, W = h->W, HD = h->HD, D = h->D, F = h->F, A = h->A, Sd = h->Sd, dt = h->dt;
    const bool b16 = h->bf16;
    Uploader up{h, w->on_device != 0};
    size_t maxe = (size_t)3 * W * W;
    if ((size_t)F * W > maxe) maxe = (size_t)F * W;
    if ((size_t)HD * W > maxe) maxe = (size_t)HD * W;
    if ((size_t)W * dt > maxe) maxe = (size_t)W * dt;
    if ((size_t)h->QKV * W > maxe) maxe = (size_t)h->QKV * W;
    if (!up.on_device || b16) JPI_TRY(dev_alloc(h, &up.tmp, maxe));

    // Small fp32 tensors.
    JPI_TRY(dev_alloc(h, &h->state_in_w, (size_t)W * Sd));
    JPI_TRY(dev_alloc(h, &h->state_in_b, W));
    JPI_TRY(dev_alloc(h, &h->action_in_w, (size_t)W * A));
    JPI_TRY(dev_alloc(h, &h->action_in_b, W));
    JPI_TRY(dev_alloc(h, &h->action_out_w, (size_t)A * W));
    JPI_TRY(dev_alloc(h, &h->action_out_b, A));
    JPI_TRY(dev_alloc(h, &h->time_in_b, W));
    JPI_TRY(dev_alloc(h, &h->time_out_b, W));
    JPI_TRY(dev_alloc(h, &h->mod_b, (size_t)mod_rows(L) * W));
    JPI_TRY(up.put(h->state_in_w, false, w->state_in_w, (size_t)W * Sd, "state_in_w"));
    JPI_TRY(up.put(h->state_in_b, false, w->state_in_b, W, "state_in_b"));
    JPI_TRY(up.put(h->action_in_w, false, w->action_in_w, (size_t)W * A, "action_in_w"));
    JPI_TRY(up.put(h->action_in_b, false, w->action_in_b, W, "action_in_b"));
    JPI_TRY(up.put(h->action_out_w, false, w->action_out_w, (size_t)A * W, "action_out_w"));
    JPI_TRY(up.put(h->action_out_b, false, w->action_out_b, A, "action_out_b"));
    JPI_TRY(up.put(h->time_in_b, false, w->time_mlp_in_b, W, "time_mlp_in_b"));
    JPI_TRY(up.put(h->time_out_b, false, w->time_mlp_out_b, W, "time_mlp_out_b"));

    // Time MLP and stacked modulation matrices in the weight type.
    const size_t ts = tw_size(h);
    JPI_TRY(dev_alloc(h, (char**)&h->time_in_w, (size_t)W * dt * ts));
    JPI_TRY(dev_alloc(h, (char**)&h->time_out_w, (size_t)W * W * ts));
    JPI_TRY(dev_alloc(h, (char**)&h->mod_w, (size_t)mod_rows(L) * W * W * ts));
    JPI_TRY(up.put(h->time_in_w, b16, w->time_mlp_in_w, (size_t)W * dt, "time_mlp_in_w"));
    JPI_TRY(up.put(h->time_out_w, b16, w->time_mlp_out_w, (size_t)W * W, "time_mlp_out_w"));
    if (!w->attn_mod_w || !w->attn_mod_b || !w->mlp_mod_w || !w->mlp_mod_b || !w->wq || !w->wk ||
        !w->wv || !w->wo || !w->w_gate || !w->w_up || !w->w_down)
        return fail(JPI_ERR_INVALID_ARG, "a per-layer weight array is NULL");
    for (int l = 0; l < L; ++l) {
        const size_t r0 = (size_t)6 * l * W;
        JPI_TRY(up.put(tw_offset(h, h->mod_w, r0 * W), b16, w->attn_mod_w[l], (size_t)3 * W * W, "attn_mod_w"));
        JPI_TRY(up.put(tw_offset(h, h->mod_w, (r0 + 3 * W) * W), b16, w->mlp_mod_w[l], (size_t)3 * W * W, "mlp_mod_w"));
        JPI_TRY(up.put(h->mod_b + r0, false, w->attn_mod_b[l], (size_t)3 * W, "attn_mod_b"));
        JPI_TRY(up.put(h->mod_b + r0 + 3 * W, false, w->mlp_mod_b[l], (size_t)3 * W, "mlp_mod_b"));
    }
    const size_t rf = (size_t)6 * L * W;
    JPI_TRY(up.put(tw_offset(h, h->mod_w, rf * W), b16, w->final_mod_w, (size_t)2 * W * W, "final_mod_w"));
    JPI_TRY(up.put(h->mod_b + rf, false, w->final_mod_b, (size_t)2 * W, "final_mod_b"));

    if (h->tc) {
        // Tensor-core path: tiled bf16 layout (tc_path.cu).
        JPI_TRY(tc_pack_layers(h, w, up.tmp, up.on_device));
    } else {
        h->plain.resize(L);
        for (int l = 0; l < L; ++l) {
            LayerPlain& p = h->plain[l];
            JPI_TRY(dev_alloc(h, (char**)&p.wqkv, (size_t)h->QKV * W * ts));
            JPI_TRY(dev_alloc(h, (char**)&p.wo, (size_t)W * HD * ts));
            JPI_TRY(dev_alloc(h, (char**)&p.wg, (size_t)F * W * ts));
            JPI_TRY(dev_alloc(h, (char**)&p.wu, (size_t)F * W * ts));
            JPI_TRY(dev_alloc(h, (char**)&p.wd, (size_t)W * F * ts));
            JPI_TRY(up.put(p.wqkv, b16, w->wq[l], (size_t)HD * W, "wq"));
            JPI_TRY(up.put(tw_offset(h, p.wqkv, (size_t)HD * W), b16, w->wk[l], (size_t)D * W, "wk"));
            JPI_TRY(up.put(tw_offset(h, p.wqkv, (size_t)(HD + D) * W), b16, w->wv[l], (size_t)D * W, "wv"));
            JPI_TRY(up.put(p.wo, b16, w->wo[l], (size_t)W * HD, "wo"));
            JPI_TRY(up.put(p.wg, b16, w->w_gate[l], (size_t)F * W, "w_gate"));
            JPI_TRY(up.put(p.wu, b16, w->w_up[l], (size_t)F * W, "w_up"));
            JPI_TRY(up.put(p.wd, b16, w->w_down[l], (size_t)W * F, "w_down"));
        }
    }
    JPI_CUDA_TRY(cudaDeviceSynchronize());
    return JPI_OK;
}

jpi_status alloc_buffers(jpi_handle* h) {
    const size_t ts = tw_size(h);
    const int W = h->W;
    const size_t Mt = (size_t)h->maxMt;
    JPI_TRY(dev_alloc(h, &h->h, Mt * W));
    JPI_TRY(dev_alloc(h, &h->x, (size_t)h->maxB * h->maxC * h->A));
    JPI_TRY(dev_alloc(h, &h->state, (size_t)h->maxB * h->Sd));
    JPI_TRY(dev_alloc(h, &h->corr, (size_t)h->maxB * JPI_MAX_CORRECTION * h->W));
    JPI_TRY(dev_alloc(h, &h->out, (size_t)h->maxB * h->maxC * h->A));
    JPI_TRY(dev_alloc(h, &h->temb, (size_t)h->maxN * h->dt));
    JPI_TRY(dev_alloc(h, &h->c1, (size_t)h->maxN * W));
    JPI_TRY(dev_alloc(h, &h->cond, (size_t)h->maxN * W));
    JPI_TRY(dev_alloc(h, &h->mods, (size_t)h->maxN * mod_rows(h->L) * W));
    const size_t actw = (size_t)(W > h->F ? W : h->F);
    JPI_TRY(dev_alloc(h, (char**)&h->act, Mt * actw * ts));
    JPI_TRY(dev_alloc(h, &h->qkv, Mt * h->QKV));
    JPI_TRY(dev_alloc(h, (char**)&h->q, Mt * h->HD * ts));
    JPI_TRY(dev_alloc(h, (char**)&h->o, Mt * h->HD * ts));
    JPI_TRY(dev_alloc(h, (char**)&h->z, Mt * h->F * ts));
    // Operand rows past a launch's last token are read by the tiled copies: start them at zero.
    JPI_CUDA_TRY(cudaMemset(h->act, 0, Mt * actw * ts));
    JPI_CUDA_TRY(cudaMemset(h->q, 0, Mt * h->HD * ts));
    JPI_CUDA_TRY(cudaMemset(h->o, 0, Mt * h->HD * ts));
    JPI_CUDA_TRY(cudaMemset(h->z, 0, Mt * h->F * ts));
    const size_t kv = (size_t)h->L * h->maxB * h->kv_rows * h->D;
    JPI_TRY(dev_alloc(h, (char**)&h->kv_k, kv * ts));
    JPI_TRY(dev_alloc(h, (char**)&h->kv_v, kv * ts));
    JPI_CUDA_TRY(cudaMemset(h->kv_k, 0, kv * ts));
    JPI_CUDA_TRY(cudaMemset(h->kv_v, 0, kv * ts));
    JPI_CUDA_TRY(cudaMemset(h->h, 0, Mt * W * sizeof(float)));
    const size_t xs_rows = (size_t)xs_tiles((int)Mt) * 64;
    JPI_TRY(dev_alloc(h, (char**)&h->hx, xs_rows * W * 2));
    JPI_CUDA_TRY(cudaMemset(h->hx, 0, xs_rows * W * 2));
    const size_t ss_slots = (size_t)((W + 127) / 128) * MAX_SPLIT_K;
    JPI_TRY(dev_alloc(h, &h->ss, ss_slots * Mt));
    JPI_CUDA_TRY(cudaMemset(h->ss, 0, ss_slots * Mt * sizeof(float)));
    JPI_TRY(dev_alloc(h, &h->dev_err, 4));
    JPI_CUDA_TRY(cudaMemset(h->dev_err, 0, 4 * sizeof(int)));
    if (h->cfg.rope_base > 0.f) {
        const int hd = h->D / 2, rows = h->maxP + h->maxS;
        std::vector<float2> tab((size_t)rows * hd);
        for (int p = 0; p < rows; ++p)
            for (int d = 0; d < hd; ++d) {
                const double ang = (double)p * std::pow((double)h->cfg.rope_base, -2.0 * d / h->D);
                tab[(size_t)p * hd + d] = make_float2((float)std::cos(ang), (float)std::sin(ang));
            }
        JPI_TRY(dev_alloc(h, &h->rope_tab, tab.size()));
        JPI_CUDA_TRY(cudaMemcpy(h->rope_tab, tab.data(), tab.size() * sizeof(float2),
                                cudaMemcpyHostToDevice));
    }
    return JPI_OK;
}

void free_handle(jpi_handle* h) {
    if (!h) return;
    cudaSetDevice(h->device);
    cudaDeviceSynchronize();
    for (auto& kv : h->graphs) cudaGraphExecDestroy(kv.second);
    h->graphs.clear();
    if (h->cap_stream) cudaStreamDestroy(h->cap_stream);
    tc_release(h);
    for (void* p : h->allocations) cudaFree(p);
    h->allocations.clear();
    cudaGetLastError();
    delete h;
}

// The whole unrolled denoise: time conditioning for every step time, then N Euler steps.
jpi_status enqueue_denoise(jpi_handle* h, int B, int C, int N, cudaStream_t st) {
    JPI_TRY(launch_time_embed(h, N, -1.0, st));
    JPI_TRY(launch_time_conditioning(h, N, st));
    const float delta = 1.0f / (float)N;
    for (int k = 0; k < N; ++k) JPI_TRY(enqueue_step(h, k, B, C, delta, nullptr, st));
    return JPI_OK;
}

jpi_status get_graph(jpi_handle* h, int B, int C, int N, cudaGraphExec_t* out) {
    const GraphKey key{B, C, N, h->cur_prefix, h->n_corr};
    auto it = h->graphs.find(key);
    if (it != h->graphs.end()) {
        *out = it->second;
        return JPI_OK;
    }
    cudaGraph_t g = nullptr;
    JPI_CUDA_TRY(cudaStreamBeginCapture(h->cap_stream, cudaStreamCaptureModeThreadLocal));
    jpi_status s = enqueue_denoise(h, B, C, N, h->cap_stream);
    cudaError_t e = cudaStreamEndCapture(h->cap_stream, &g);
    if (s != JPI_OK) {
        if (g) cudaGraphDestroy(g);
        return s;
    }
    if (e != cudaSuccess) return fail(JPI_ERR_CUDA, "graph capture failed: %s", cudaGetErrorString(e));
    cudaGraphExec_t ex = nullptr;
    e = cudaGraphInstantiate(&ex, g, 0);
    if (e != cudaSuccess) {
        cudaGraphDestroy(g);
        return fail(JPI_ERR_CUDA, "graph instantiate failed: %s", cudaGetErrorString(e));
    }
    size_t n = 0;
    int kernels = 0;
    if (cudaGraphGetNodes(g, nullptr, &n) == cudaSuccess && n) {
        std::vector<cudaGraphNode_t> nodes(n);
        if (cudaGraphGetNodes(g, nodes.data(), &n) == cudaSuccess)
            for (auto nd : nodes) {
                cudaGraphNodeType t;
                if (cudaGraphNodeGetType(nd, &t) == cudaSuccess && t == cudaGraphNodeTypeKernel) ++kernels;
            }
    }
    cudaGraphDestroy(g);
    h->graph_kernels[key] = kernels;
    h->graphs[key] = ex;
    *out = ex;
    return JPI_OK;
}

}  // namespace

// One Euler step (or one forward): token embedding, L layers, final norm + projection.
jpi_status enqueue_step(jpi_handle* h, int step, int B, int C, float delta, float* v_out,
                        cudaStream_t st) {
    JPI_TRY(launch_embed(h, step, B, C, h->x, st));
    for (int l = 0; l < h->L; ++l) {
        if (h->tc)
            JPI_TRY(tc_launch_layer(h, l, step, B, C, st));
        else
            JPI_TRY(launch_layer_simt(h, l, step, B, C, st));
    }
    return launch_final(h, step, B, C, delta, v_out ? nullptr : h->x, v_out, nullptr, st);
}

jpi_status check_call(jpi_handle* h, int B, int C, int N) {
    if (!h) return fail(JPI_ERR_INVALID_ARG, "handle is NULL");
    if (B < 1 || C < 1 || N < 1) return fail(JPI_ERR_INVALID_ARG, "batch, chunk and num_steps must be >= 1");
    if (B > h->maxB || C > h->maxC || N > h->maxN)
        return fail(JPI_ERR_SHAPE, "batch %d / chunk %d / steps %d exceed the maxima %d / %d / %d",
                    B, C, N, h->maxB, h->maxC, h->maxN);
    if (!h->prefix_ready) return fail(JPI_ERR_NOT_READY, "no prefix KV has been set");
    if (B != h->cur_batch)
        return fail(JPI_ERR_SHAPE, "batch %d differs from the prefix KV's batch %d", B, h->cur_batch);
    if (h->n_corr > 0 && B != h->corr_batch)
        return fail(JPI_ERR_SHAPE, "batch %d differs from the correction items' batch %d", B, h->corr_batch);
    return JPI_OK;
}

}  // namespace jpi

using namespace jpi;

extern "C" {

JPI_API const char* jpi_last_error(void) { return g_err; }

JPI_API jpi_status jpi_expert_create(const jpi_config* cfg, const jpi_weights* w, jpi_handle** out) {
    clear_error();
    if (!out) return fail(JPI_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    JPI_TRY(check_config(cfg));
    if (!w) return fail(JPI_ERR_INVALID_ARG, "weights are NULL");
    jpi_handle* h = new (std::nothrow) jpi_handle();
    if (!h) return fail(JPI_ERR_OOM, "host allocation failed");
    h->cfg = *cfg;
    h->bf16 = cfg->precision == JPI_BF16;
    h->L = cfg->n_layers; h->W = cfg->width; h->H = cfg->n_heads; h->D = cfg->head_dim;
    h->F = cfg->mlp_dim; h->A = cfg->action_dim; h->Sd = cfg->state_dim; h->dt = cfg->time_dim;
    h->HD = h->H * h->D; h->QKV = (h->H + 2) * h->D;
    h->maxB = cfg->max_batch; h->maxP = cfg->max_prefix; h->maxC = cfg->max_chunk;
    h->maxS = cfg->max_chunk + 1 + JPI_MAX_CORRECTION; h->maxN = cfg->max_steps;
    h->maxMt = h->maxB * h->maxS;
    h->kv_rows = h->maxP + h->maxS;
    jpi_status s = JPI_OK;
    cudaError_t e = cudaGetDevice(&h->device);
    if (e != cudaSuccess) {
        delete h;
        return fail(JPI_ERR_CUDA, "no CUDA device: %s", cudaGetErrorString(e));
    }
    h->tc = h->bf16 && tc_supported(h);
    if ((s = alloc_buffers(h)) != JPI_OK || (s = pack_weights(h, w)) != JPI_OK ||
        (s = configure_simt_kernels(h)) != JPI_OK || (h->tc && (s = tc_prepare(h)) != JPI_OK)) {
        std::string msg = g_err;
        free_handle(h);
        return fail(s, "%s", msg.c_str());
    }
    e = cudaStreamCreateWithFlags(&h->cap_stream, cudaStreamNonBlocking);
    if (e != cudaSuccess) {
        free_handle(h);
        return fail(JPI_ERR_CUDA, "stream creation failed: %s", cudaGetErrorString(e));
    }
    *out = h;
    return JPI_OK;
}

JPI_API jpi_status jpi_expert_destroy(jpi_handle* h) {
    clear_error();
    free_handle(h);
    return JPI_OK;
}

JPI_API jpi_status jpi_set_prefix_kv(jpi_handle* h, const void* const* k_layers,
                                     const void* const* v_layers, int batch, int prefix_len,
                                     int kv_is_fp32, void* stream) {
    clear_error();
    if (!h || !k_layers || !v_layers) return fail(JPI_ERR_INVALID_ARG, "NULL handle or layer arrays");
    if (batch < 1 || prefix_len < 1) return fail(JPI_ERR_INVALID_ARG, "batch and prefix_len must be >= 1");
    if (batch > h->maxB || prefix_len > h->maxP)
        return fail(JPI_ERR_SHAPE, "batch %d / prefix %d exceed the maxima %d / %d", batch,
                    prefix_len, h->maxB, h->maxP);
    for (int l = 0; l < h->L; ++l)
        if (!k_layers[l] || !v_layers[l]) return fail(JPI_ERR_INVALID_ARG, "layer %d K or V is NULL", l);
    cudaStream_t st = (cudaStream_t)stream;
    const size_t layer_elems = (size_t)h->maxB * h->kv_rows * h->D;
    for (int l = 0; l < h->L; ++l) {
        JPI_TRY(launch_convert_kv(h, k_layers[l], kv_is_fp32, tw_offset(h, h->kv_k, l * layer_elems),
                                  batch, prefix_len, st));
        JPI_TRY(launch_convert_kv(h, v_layers[l], kv_is_fp32, tw_offset(h, h->kv_v, l * layer_elems),
                                  batch, prefix_len, st));
    }
    h->cur_batch = batch;
    h->cur_prefix = prefix_len;
    h->prefix_ready = true;
    return JPI_OK;
}

JPI_API jpi_status jpi_prefix_kv_ptr(jpi_handle* h, int layer, void** k, void** v,
                                     long long* request_stride) {
    clear_error();
    if (!h || !k || !v || !request_stride) return fail(JPI_ERR_INVALID_ARG, "NULL argument");
    if (layer < 0 || layer >= h->L) return fail(JPI_ERR_INVALID_ARG, "layer %d out of range", layer);
    const size_t layer_elems = (size_t)h->maxB * h->kv_rows * h->D;
    *k = tw_offset(h, h->kv_k, layer * layer_elems);
    *v = tw_offset(h, h->kv_v, layer * layer_elems);
    *request_stride = (long long)h->kv_rows * h->D;
    return JPI_OK;
}

JPI_API jpi_status jpi_commit_prefix(jpi_handle* h, int batch, int prefix_len) {
    clear_error();
    if (!h) return fail(JPI_ERR_INVALID_ARG, "handle is NULL");
    if (batch < 1 || prefix_len < 1) return fail(JPI_ERR_INVALID_ARG, "batch and prefix_len must be >= 1");
    if (batch > h->maxB || prefix_len > h->maxP) return fail(JPI_ERR_SHAPE, "batch/prefix exceed the maxima");
    h->cur_batch = batch;
    h->cur_prefix = prefix_len;
    h->prefix_ready = true;
    return JPI_OK;
}

JPI_API jpi_status jpi_set_correction(jpi_handle* h, const float* items, int batch, int num_items,
                                      void* stream) {
    clear_error();
    if (!h) return fail(JPI_ERR_INVALID_ARG, "handle is NULL");
    if (num_items < 0 || batch < 1) return fail(JPI_ERR_INVALID_ARG, "num_items must be >= 0 and batch >= 1");
    if (num_items > JPI_MAX_CORRECTION || batch > h->maxB)
        return fail(JPI_ERR_SHAPE, "num_items %d / batch %d exceed the maxima %d / %d", num_items, batch,
                    JPI_MAX_CORRECTION, h->maxB);
    if (num_items > 0 && !items) return fail(JPI_ERR_INVALID_ARG, "items are NULL");
    if (num_items > 0)
        JPI_CUDA_TRY(cudaMemcpyAsync(h->corr, items, (size_t)batch * num_items * h->W * sizeof(float),
                                     cudaMemcpyDeviceToDevice, (cudaStream_t)stream));
    h->n_corr = num_items;
    h->corr_batch = batch;
    return JPI_OK;
}

JPI_API jpi_status jpi_denoise(jpi_handle* h, const float* state, const float* noise, int batch,
                               int chunk, int num_steps, float* out_actions, void* stream) {
    clear_error();
    JPI_TRY(check_call(h, batch, chunk, num_steps));
    if (!state || !noise || !out_actions) return fail(JPI_ERR_INVALID_ARG, "NULL input or output");
    cudaStream_t st = (cudaStream_t)stream;
    cudaGraphExec_t ex = nullptr;
    JPI_TRY(get_graph(h, batch, chunk, num_steps, &ex));
    const size_t nx = (size_t)batch * chunk * h->A;
    JPI_CUDA_TRY(cudaMemcpyAsync(h->state, state, (size_t)batch * h->Sd * sizeof(float),
                                 cudaMemcpyDeviceToDevice, st));
    JPI_CUDA_TRY(cudaMemcpyAsync(h->x, noise, nx * sizeof(float), cudaMemcpyDeviceToDevice, st));
    JPI_CUDA_TRY(cudaGraphLaunch(ex, st));
    JPI_CUDA_TRY(cudaMemcpyAsync(out_actions, h->x, nx * sizeof(float), cudaMemcpyDeviceToDevice, st));
    return JPI_OK;
}

JPI_API jpi_status jpi_denoise_host(jpi_handle* h, const float* state, const float* noise,
                                    int batch, int chunk, int num_steps, float* out_actions,
                                    void* stream) {
    clear_error();
    JPI_TRY(check_call(h, batch, chunk, num_steps));
    if (!state || !noise || !out_actions) return fail(JPI_ERR_INVALID_ARG, "NULL input or output");
    cudaStream_t st = (cudaStream_t)stream;
    cudaGraphExec_t ex = nullptr;
    JPI_TRY(get_graph(h, batch, chunk, num_steps, &ex));
    const size_t nx = (size_t)batch * chunk * h->A;
    JPI_CUDA_TRY(cudaMemcpyAsync(h->state, state, (size_t)batch * h->Sd * sizeof(float),
                                 cudaMemcpyHostToDevice, st));
    JPI_CUDA_TRY(cudaMemcpyAsync(h->x, noise, nx * sizeof(float), cudaMemcpyHostToDevice, st));
    JPI_CUDA_TRY(cudaGraphLaunch(ex, st));
    JPI_CUDA_TRY(cudaMemcpyAsync(out_actions, h->x, nx * sizeof(float), cudaMemcpyDeviceToHost, st));
    JPI_CUDA_TRY(cudaStreamSynchronize(st));
    return JPI_OK;
}

JPI_API jpi_status jpi_expert_forward(jpi_handle* h, const float* state, const float* x_t, float t,
                                      int batch, int chunk, float* out_v, float* out_h,
                                      void* stream) {
    clear_error();
    JPI_TRY(check_call(h, batch, chunk, 1));
    if (!state || !x_t || !out_v) return fail(JPI_ERR_INVALID_ARG, "NULL input or output");
    if (!(t >= 0.f)) return fail(JPI_ERR_INVALID_ARG, "t must be >= 0");
    cudaStream_t st = (cudaStream_t)stream;
    JPI_CUDA_TRY(cudaMemcpyAsync(h->state, state, (size_t)batch * h->Sd * sizeof(float),
                                 cudaMemcpyDeviceToDevice, st));
    JPI_CUDA_TRY(cudaMemcpyAsync(h->x, x_t, (size_t)batch * chunk * h->A * sizeof(float),
                                 cudaMemcpyDeviceToDevice, st));
    JPI_TRY(launch_time_embed(h, 1, (double)t, st));
    JPI_TRY(launch_time_conditioning(h, 1, st));
    JPI_TRY(enqueue_step(h, 0, batch, chunk, 0.f, out_v, st));
    if (out_h)
        JPI_CUDA_TRY(cudaMemcpyAsync(out_h, h->h, (size_t)batch * (chunk + h->n_ctx()) * h->W * sizeof(float),
                                     cudaMemcpyDeviceToDevice, st));
    return JPI_OK;
}

JPI_API jpi_status jpi_device_status(jpi_handle* h) {
    clear_error();
    if (!h) return fail(JPI_ERR_INVALID_ARG, "handle is NULL");
    JPI_CUDA_TRY(cudaDeviceSynchronize());
    int err = 0;
    JPI_CUDA_TRY(cudaMemcpy(&err, h->dev_err, sizeof(int), cudaMemcpyDeviceToHost));
    if (err != DEV_OK) {
        JPI_CUDA_TRY(cudaMemset(h->dev_err, 0, sizeof(int)));
        return fail(JPI_ERR_DEVICE_TIMEOUT, "device-side error code %d (bounded wait gave up)", err);
    }
    return JPI_OK;
}

JPI_API jpi_status jpi_graph_kernel_count(jpi_handle* h, int batch, int chunk, int num_steps,
                                          int* count) {
    clear_error();
    JPI_TRY(check_call(h, batch, chunk, num_steps));
    if (!count) return fail(JPI_ERR_INVALID_ARG, "count is NULL");
    cudaGraphExec_t ex = nullptr;
    JPI_TRY(get_graph(h, batch, chunk, num_steps, &ex));
    *count = h->graph_kernels[GraphKey{batch, chunk, num_steps, h->cur_prefix, h->n_corr}];
    return JPI_OK;
}

JPI_API jpi_status jpi_profile_op(jpi_handle* h, int op, int layer, int batch, int chunk,
                                  int num_steps, int reps, void* stream) {
    clear_error();
    JPI_TRY(check_call(h, batch, chunk, num_steps));
    if (op < 0 || op > 7 || layer < 0 || layer >= h->L || reps < 1)
        return fail(JPI_ERR_INVALID_ARG, "bad op %d / layer %d / reps %d", op, layer, reps);
    cudaStream_t st = (cudaStream_t)stream;
    for (int r = 0; r < reps; ++r) {
        switch (op) {
            case 0:
                JPI_TRY(launch_time_embed(h, num_steps, -1.0, st));
                JPI_TRY(launch_time_conditioning(h, num_steps, st));
                break;
            case 1: JPI_TRY(launch_embed(h, 0, batch, chunk, h->x, st)); break;
            case 7:
                JPI_TRY(launch_final(h, 0, batch, chunk, 0.f, nullptr, h->out, nullptr, st));
                break;
            default:
                if (h->tc)
                    JPI_TRY(tc_launch_op(h, op, layer, 0, batch, chunk, st));
                else
                    JPI_TRY(launch_op_simt(h, op, layer, 0, batch, chunk, st));
        }
    }
    return JPI_OK;
}

JPI_API jpi_status jpi_memory_usage(const jpi_handle* h, long long* bytes) {
    clear_error();
    if (!h || !bytes) return fail(JPI_ERR_INVALID_ARG, "NULL argument");
    *bytes = (long long)h->device_bytes;
    return JPI_OK;
}

}  // extern "C"
