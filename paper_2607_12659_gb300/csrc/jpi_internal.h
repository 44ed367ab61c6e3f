// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cstdint>
#include <cstddef>
#include <map>
#include <string>
#include <tuple>
#include <vector>

#include "jpi.h"

namespace jpi {

// Last-error message of the calling host thread.
void set_error(const char* fmt, ...);
void clear_error();

#define JPI_CUDA_TRY(expr)                                                        \
    do {                                                                          \
        cudaError_t e_ = (expr);                                                  \
        if (e_ != cudaSuccess) {                                                  \
            ::jpi::set_error("%s failed: %s (%s:%d)", #expr, cudaGetErrorString(e_), \
                             __FILE__, __LINE__);                                 \
            return JPI_ERR_CUDA;                                                  \
        }                                                                         \
    } while (0)

#define JPI_TRY(expr)                        \
    do {                                     \
        jpi_status s_ = (expr);              \
        if (s_ != JPI_OK) return s_;         \
    } while (0)

// Device error codes written by bounded waits inside kernels (first writer wins).
enum DeviceError : int {
    DEV_OK = 0,
    DEV_TIMEOUT_WEIGHTS = 1,   // weight tile TMA never completed
    DEV_TIMEOUT_MMA = 2,       // tensor-core commit never arrived
    DEV_BAD_SHAPE = 3,         // a kernel saw a shape it cannot tile
    DEV_FP16_RANGE = 4,        // a residual-stream value exceeded the fp16 range of its copy
};

// Offsets (in rows of W) of the modulation vectors inside one step's modulation row block.
// Layer l: attention (sigma, beta, gamma) at 6 l + {0,1,2}, MLP at 6 l + {3,4,5};
// the final norm's (sigma, beta) at 6 L + {0, 1}.
inline int mod_rows(int L) { return 6 * L + 2; }

// Largest split of a projection's K range over the CTAs of a cluster. The per-token sums of
// squares of the residual stream are kept in up to (W / 128) x MAX_SPLIT_K slots.
constexpr int MAX_SPLIT_K = 16;

// Operand of the RMSNorm-fed projections on the tensor-core path: xs = bf16((1 + sigma) * h) for
// the next norm's scale sigma, in tiles of 64 rows: 63 token rows, then one row holding the
// norm's shift beta. The projection of a tile then carries W * beta in its last column, and the
// per-token 1 / rms(h) is applied to the product: W u = rinv * (W xs) + W beta for the adaptive
// RMSNorm u = h * rinv * (1 + sigma) + beta of App. A's expert layers.
constexpr int XS_TOKENS = 63;
__host__ __device__ inline int xs_row(int t) { return (t / XS_TOKENS) * 64 + t % XS_TOKENS; }
__host__ __device__ inline int xs_tiles(int Mt) { return (Mt + XS_TOKENS - 1) / XS_TOKENS; }

// Plain (un-tiled) layer weights used by the CUDA-core kernels.
struct LayerPlain {
    void* wqkv;   // [(H+2) D][W]: rows of wq, then wk, then wv
    void* wo;     // [W][H D]
    void* wg;     // [F][W]
    void* wu;     // [F][W]
    void* wd;     // [W][F]
};

// Tensor-core (tcgen05) layer weights: tiles of 128 rows x 64 K-elements (16 KiB of bf16),
// stored tile-contiguously in [row tile][k block] order so that one bulk tensor copy moves one
// contiguous tile. Row order inside the QKV and gate/up matrices is permuted so that the rows
// an epilogue pairs (the two halves of a rotary pair, or a gate row and its up row) sit in
// rows r and r + 64 of the same tile.
struct LayerTiled {
    __nv_bfloat16* qkv;    // [(H+2) D / 128 tiles][W / 64][128][64]
    __nv_bfloat16* o;      // [W / 128][H D / 64][128][64]
    __nv_bfloat16* gu;     // [2 F / 128][W / 64][128][64]
    __nv_bfloat16* down;   // [W / 128][F / 64][128][64]
};

// Work split of one tensor-core projection: `ntiles` 128-row weight tiles, each reduced over
// K by a cluster of `splits` CTAs that own `kpb` 64-wide K blocks apiece.
struct GemmPlan {
    int rows = 0, K = 0, ntiles = 0, nkb = 0, kpb = 0, splits = 0, ctas = 0;
    size_t smem = 0;
};

struct GraphKey {
    int batch, chunk, steps, prefix, items;
    bool operator<(const GraphKey& o) const {
        return std::tie(batch, chunk, steps, prefix, items) < std::tie(o.batch, o.chunk, o.steps, o.prefix, o.items);
    }
};

}  // namespace jpi

struct jpi_handle {
    jpi_config cfg;
    int device = 0;
    bool bf16 = true;
    bool tc = false;          // tensor-core kernels in use (bf16 mode with supported dims)
    bool pdl = true;          // programmatic dependent launch between tensor-core kernels
    int num_sms = 0;
    int attn_max_splits = 8;  // largest key-split cluster of the attention kernel
    int attn_force_splits = 0;  // > 0: key splits asked of the split-KV attention (JPI_ATTN_SPLITS)
    bool batch_invariant = false;   // kernels and splits of one request at every batch size (JPI_BATCH_INVARIANT)

    // Dimensions.
    int L, W, H, D, F, A, Sd, dt, HD, QKV;   // QKV = (H + 2) D
    int maxB, maxP, maxC, maxS, maxN, maxMt, kv_rows;

    // ---- Device memory (all allocated in create) ----
    std::vector<void*> allocations;
    size_t device_bytes = 0;

    // Weights. Element type is bf16 in JPI_BF16 mode, fp32 in JPI_FP32 mode ("TW").
    std::vector<jpi::LayerPlain> plain;
    std::vector<jpi::LayerTiled> tiled;
    void* mod_w = nullptr;       // [(6L+2) W][W] TW, all modulation matrices stacked
    float* mod_b = nullptr;      // [(6L+2) W]
    void* time_in_w = nullptr;   // [W][d_t] TW
    float* time_in_b = nullptr;  // [W]
    void* time_out_w = nullptr;  // [W][W] TW
    float* time_out_b = nullptr; // [W]
    float* state_in_w = nullptr; // [W][S_d] fp32
    float* state_in_b = nullptr;
    float* action_in_w = nullptr;   // [W][A] fp32
    float* action_in_b = nullptr;
    float* action_out_w = nullptr;  // [A][W] fp32
    float* action_out_b = nullptr;
    float2* rope_tab = nullptr;     // [maxP + maxS][D/2] (cos, sin); null when rope_base == 0

    // KV store: [L][maxB][kv_rows][D], element type TW; rows 0..P-1 prefix, P..P+S-1 suffix.
    void* kv_k = nullptr;
    void* kv_v = nullptr;

    // Activations.
    float* h = nullptr;         // [maxMt][W] residual stream
    float* x = nullptr;         // [maxB][maxC][A] current actions
    float* state = nullptr;     // [maxB][S_d] staged state
    float* out = nullptr;       // [maxB][maxC][A] staged output
    float* temb = nullptr;      // [maxN][d_t] time embeddings
    float* c1 = nullptr;        // [maxN][W]
    float* cond = nullptr;      // [maxN][W]
    float* mods = nullptr;      // [maxN][(6L+2) W]
    void* act = nullptr;        // [maxMt][max(W, F)] GEMM input (TW type)
    float* qkv = nullptr;       // [maxMt][QKV] raw projections (CUDA-core path)
    void* q = nullptr;          // [maxMt][H][D] rotated queries (TW type)
    void* o = nullptr;          // [maxMt][H D] attention output (TW type)
    void* z = nullptr;          // [maxMt][F] GeGLU output (TW type)
    float* ss = nullptr;        // [W / 128][maxMt] per-token sums of h^2 over 128-feature slices
    void* hx = nullptr;         // [xs_tiles(maxMt) x 64][W] bf16 scaled h (+ beta rows), see xs_row
    int* dev_err = nullptr;     // device error word

    // Tensor-core path: one plan per projection (QKV, O, gate/up, down) and tensor maps
    // (4 per layer, same order).
    jpi::GemmPlan plans[4];
    int big_min_tokens[4] = {512, 128, 128, 128};   // per projection kind: from this many tokens the large-M GEMM
    int big_split = 0;          // K split of the large-M residual projections (0: chosen per launch)
    int big_clusters[4] = {0, 0, 0, 0};   // co-resident large-M clusters of 1, 2, 4, 8 CTAs
    int attn_t5_min_batch = 3;  // batches of at least this many requests use the tcgen05 attention
    bool attn_t5 = false;       // its tensor maps and attributes are ready
    int attn_t5_splits = 0;     // its key split (0: chosen per launch)
    int t5_clusters[5] = {};    // co-resident clusters of s CTAs of it, s = 1..4
    void* t5_ws = nullptr;      // its key-split workspace: partial outputs, then (m, l)
    void* t5_wml = nullptr;
    CUtensorMap amaps[3];       // attention operands: q, prefix/suffix K, V (all layers)
    CUtensorMap qmap_at;        // q as 32-row boxes for the split-KV attention
    CUtensorMap kmap_at, vmap_at;   // K, V of all layers as 32-row boxes for it
    std::vector<CUtensorMap> tmaps;
    bool mod_tc = false;        // modulation vectors on tensor cores (mod_tc.cu)
    CUtensorMap mod_map;        // the stacked modulation matrix [(6L+2) W][W] as 128 x 64 boxes
    CUtensorMap xmaps[3];       // B operands: hx, o, z

    // State.
    int cur_batch = 0, cur_prefix = 0;
    bool prefix_ready = false;
    // Correction items (context tokens after the state token): [maxB][JPI_MAX_CORRECTION][W] fp32,
    // n_corr of them per request for corr_batch requests. Suffix rows 0 .. n_ctx() - 1 are the
    // state and context tokens, then the actions.
    float* corr = nullptr;
    int n_corr = 0, corr_batch = 0;
    int n_ctx() const { return 1 + n_corr; }
    cudaStream_t cap_stream = nullptr;
    std::map<jpi::GraphKey, cudaGraphExec_t> graphs;
    std::map<jpi::GraphKey, int> graph_kernels;
};

namespace jpi {

// Kernel launchers (kernels_simt.cu). All enqueue on `st` and return JPI_OK or JPI_ERR_CUDA.
jpi_status configure_simt_kernels(jpi_handle* h);
jpi_status launch_time_embed(jpi_handle* h, int nsteps, double t_override, cudaStream_t st);
jpi_status launch_time_conditioning(jpi_handle* h, int nsteps, cudaStream_t st);
jpi_status launch_time_conditioning_into(jpi_handle* h, double t, float* temb, float* c1,
                                         float* cond, cudaStream_t st);
jpi_status launch_embed(jpi_handle* h, int step, int batch, int chunk, const float* x, cudaStream_t st);
jpi_status launch_layer_simt(jpi_handle* h, int layer, int step, int batch, int chunk,
                             cudaStream_t st);
// One sub-step of a layer (ops 2..6 of jpi_profile_op).
jpi_status launch_op_simt(jpi_handle* h, int op, int layer, int step, int batch, int chunk,
                          cudaStream_t st);
jpi_status launch_final(jpi_handle* h, int step, int batch, int chunk, float delta,
                        float* x_inout, float* v_out, float* out_copy, cudaStream_t st);
jpi_status launch_convert_kv(jpi_handle* h, const void* src, int src_fp32, void* dst,
                             int batch, int prefix_len, cudaStream_t st);

// Entry-point helpers (api.cu). check_call: host-side checks of a denoise or forward call of
// `B` requests, `C` actions and `N` steps against the handle's maxima, its prefix and its
// correction items. enqueue_step: one Euler step (or, with v_out set, one forward pass) from
// the modulation vectors of step slot `step`: token embedding, the L layers, final norm and
// projection.
jpi_status check_call(jpi_handle* h, int B, int C, int N);
jpi_status enqueue_step(jpi_handle* h, int step, int B, int C, float delta, float* v_out,
                        cudaStream_t st);

}  // namespace jpi
