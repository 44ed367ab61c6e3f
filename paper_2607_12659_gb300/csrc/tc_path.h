// Tensor-core (tcgen05 + TMA) path of the bf16 expert layers.
#pragma once
#include "jpi_internal.h"

namespace jpi {

// True when the handle's dimensions are tiled by the tensor-core kernels.
bool tc_supported(const jpi_handle* h);
// Packs the per-layer projection/MLP matrices into the tiled bf16 layout (see LayerTiled).
jpi_status tc_pack_layers(jpi_handle* h, const jpi_weights* w, float* tmp, bool on_device);
// Builds tensor maps, workspaces and kernel attributes once the buffers exist.
jpi_status tc_prepare(jpi_handle* h);
// Enqueues one expert layer (norm + QKV + rotary, attention, O-proj, norm + GeGLU, down).
jpi_status tc_launch_layer(jpi_handle* h, int layer, int step, int batch, int chunk,
                           cudaStream_t st);
// One sub-step of a layer (ops 2..6 of jpi_profile_op).
jpi_status tc_launch_op(jpi_handle* h, int op, int layer, int step, int batch, int chunk,
                        cudaStream_t st);
// Tensor-core attention (attn_tc.cu).
bool attn_tc_supported(const jpi_handle* h);
jpi_status attn_tc_prepare(jpi_handle* h);
jpi_status launch_attn_tc(jpi_handle* h, int layer, int batch, int chunk, cudaStream_t st);
// Tensor-core attention without key splits for batched launches (attn_t5.cu).
bool attn_t5_supported(const jpi_handle* h);
jpi_status attn_t5_prepare(jpi_handle* h);
jpi_status launch_attn_t5(jpi_handle* h, int layer, int batch, int chunk, cudaStream_t st);
// Modulation vectors of N <= 16 step times on tensor cores (mod_tc.cu): Y [N][(6L+2) W] from
// X [N][W]; used in bf16 mode when mod_tc_prepare set h->mod_tc.
bool mod_tc_supported(const jpi_handle* h);
jpi_status mod_tc_prepare(jpi_handle* h);
jpi_status launch_mod_tc(jpi_handle* h, const float* X, float* Y, int N, cudaStream_t st);
// 2D bf16 tensor map over [rows][cols] row-major, 128-byte swizzle, box {64 cols, box_rows}.
jpi_status tc_make_tmap(const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows, CUtensorMap* map);
// Frees what tc_prepare created outside the handle's allocation list.
void tc_release(jpi_handle* h);

}  // namespace jpi
