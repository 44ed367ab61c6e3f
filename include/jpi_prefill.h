/*
 * jpi_prefill.h — C-ABI of the VLM's LLM prefill that fills the action expert's KV store.
 *
 * Paper passages this interface follows:
 *   - App. A ("Model Architecture of pi series Models") and Tab. "Model architecture parameters
 *     of pi series VLA models": the LLM (Gemma 2B: 18 layers, width 2048, 8 heads of 256)
 *     processes the image and language tokens, and each of its layers hands its KV cache to the
 *     matching layer of the action expert.
 *   - Sec. 4.3 ("System Design"): the intermediate buffers between the components stay on the
 *     GPU. The prefill writes every layer's rotated keys and values straight into the expert's
 *     store (the zero-copy producer path of jpi_prefix_kv_ptr / jpi_commit_prefix in jpi.h).
 * The paper leaves the block's details open; this library and its CPU reference read them as:
 * one KV head of width head_dim shared by all query heads; pre-norm Gemma blocks without biases,
 * h += Wo attn(RMSNorm(h) (1 + a)), h += Wd (gelu_tanh(Wg u) * (Wu u)) with u = RMSNorm(h) (1 + m);
 * rotary coding (rotate-half, base rope_base) of queries and keys at positions 0 .. P-1, the
 * rotated keys cached; every prefix token attends to every prefix token; the final output is
 * RMSNorm(h) (1 + final_norm), the VLM state the correction module's compressor reads.
 *
 * Built as its own library (libjpi_prefill.so): its products are plain bf16 GEMMs of
 * batch * prefix rows, which run on its own tcgen05 tensor-core kernel with fp32 accumulation
 * (no library GEMM); norms, rotary coding, softmax and GeGLU run in its own kernels. Conventions
 * are those of jpi.h (status codes, host-side checks before anything is enqueued, row-major
 * [out][in] matrices, one host thread and one stream per handle), with its own
 * jpi_prefill_last_error().
 */
#ifndef JPI_PREFILL_H
#define JPI_PREFILL_H

#include "jpi.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct jpi_prefill_handle jpi_prefill_handle;

typedef struct jpi_prefill_config {
    int n_layers;     /* L (18)                                                                   */
    int width;        /* W, residual width (2048); a multiple of 8                                */
    int n_heads;      /* H query heads (8); one shared KV head                                    */
    int head_dim;     /* D (256), also the KV width; even, a multiple of 8, at most 512           */
    int mlp_dim;      /* F, GeGLU width (16384); a multiple of 8                                  */
    int max_batch;    /* most requests per call                                                   */
    int max_prefix;   /* most prefix tokens per request                                           */
    float rope_base;  /* 10000; 0 disables rotary coding                                          */
    float rms_eps;    /* 1e-6                                                                     */
} jpi_prefill_config;

/* fp32 weights, host or device (on_device); create rounds the matrices to bf16 (nearest even).
 * Per-layer tensors are arrays of L pointers. Norm scales w enter as (1 + w). */
typedef struct jpi_prefill_weights {
    const float* const* attn_norm;   /* [W]                                                      */
    const float* const* wq;          /* [H D][W]                                                 */
    const float* const* wk;          /* [D][W]                                                   */
    const float* const* wv;          /* [D][W]                                                   */
    const float* const* wo;          /* [W][H D]                                                 */
    const float* const* mlp_norm;    /* [W]                                                      */
    const float* const* w_gate;      /* [F][W]                                                   */
    const float* const* w_up;        /* [F][W]                                                   */
    const float* const* w_down;      /* [W][F]                                                   */
    const float* final_norm;         /* [W]                                                      */
    int on_device;
} jpi_prefill_weights;

/* Creates a handle: checks the shapes, packs the weights as bf16 and allocates every buffer for
 * the maxima. Synchronous. On failure *out is NULL. */
JPI_API jpi_status jpi_prefill_create(const jpi_prefill_config* cfg, const jpi_prefill_weights* w,
                                      jpi_prefill_handle** out);
JPI_API jpi_status jpi_prefill_destroy(jpi_prefill_handle* h);   /* NULL is a no-op */

/*
 * Runs the prefill of `batch` requests of `prefix_len` tokens each.
 *   x:          device [batch][prefix_len][W] token embeddings, fp32 (x_is_fp32 = 1) or bf16.
 *   k_layers[l], v_layers[l]: device bf16 destinations of layer l's rotated keys and values:
 *               request b's row p, element d at base + b * request_stride + p * D + d (elements),
 *               exactly what jpi_prefix_kv_ptr returns for a JPI_BF16 expert handle. Both arrays
 *               are host arrays of L device pointers.
 *   out_final:  device [batch][prefix_len][W] fp32, the final-layer output, or NULL.
 * 1 <= batch <= max_batch, 1 <= prefix_len <= max_prefix, request_stride >= prefix_len * D.
 * Enqueued on `stream`; the inputs must stay valid until the stream reaches the call. After it,
 * jpi_commit_prefix(expert, batch, prefix_len) makes the store current for the expert.
 */
JPI_API jpi_status jpi_prefill_run(jpi_prefill_handle* h, const void* x, int x_is_fp32, int batch,
                                   int prefix_len, void* const* k_layers, void* const* v_layers,
                                   long long request_stride, float* out_final, void* stream);

/*
 * Synchronises the device and reports device-side errors of earlier runs: JPI_OK, or
 * JPI_ERR_DEVICE_TIMEOUT if a bounded wait inside a product kernel gave up (that kernel skipped
 * its stores and returned; the outputs of that run are invalid; the word is cleared), or
 * JPI_ERR_CUDA.
 */
JPI_API jpi_status jpi_prefill_device_status(jpi_prefill_handle* h);

JPI_API jpi_status jpi_prefill_memory_usage(const jpi_prefill_handle* h, long long* bytes);
JPI_API const char* jpi_prefill_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* JPI_PREFILL_H */
