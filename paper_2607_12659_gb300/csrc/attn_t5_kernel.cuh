// The tcgen05 suffix/prefix attention kernel, shared by the expert (csrc/attn_t5.cu) and the LLM
// prefill (csrc/prefill/prefill.cu); each library includes it once, inside its own translation
// unit. Its device error codes: T5_ERR_LOAD (a K/V bulk copy never completed), T5_ERR_MMA (a
// tensor-core commit never arrived).
//
// App. A of the paper: the expert's queries (state token + C action tokens, all H heads) attend
// over the matching LLM layer's KV cache followed by the suffix's own keys/values; one KV head
// is shared by all heads, so one request is a dense [S*H] x [P+S] problem (rows token-major,
// row = i * H + head; the state row i = 0 and the correction items' context rows i < nctx see
// the prefix and each other only).
//
// One CTA = 128 query rows of one request over all of its keys, in blocks of 64 keys (two TMEM
// score buffers and two shared-memory P buffers, so block i+1's softmax overlaps block i's P V):
//   warp 0  one thread: bulk tensor copies of the query tile once, then K blocks through a
//           two-slot ring (K of block i+2 as soon as S_i is done);
//   warp 1  one thread: V blocks through a two-slot ring of their own (V of block i+2 once
//           P_i V_i is done); prefix blocks of either may be fetched before the dependency wait;
//   warp 2  one thread: S_i = Q K_i^T (M = 128, N = 64, K = D) into one of two TMEM score
//           buffers: S_0, S_1, then S_{i+2} as soon as P_i is written (its score buffer is free);
//   warp 3  one thread: O += P_i V_i (M = 128, N = D, K = 64) into the TMEM output with V read
//           as an MN-major operand straight from its bulk copy, as soon as P_i and V_i are in.
//           The two MMA chains are issued by two threads, so neither waits on the other's issue
//           (one thread issues an N = 64 MMA every ~50-75 cycles, longer than it runs);
//   warps 4-7  one query row per thread (its TMEM lane): scale, mask, block maximum, softmax
//           probabilities P_i written to shared memory (bf16, 128-byte swizzled K-major rows).
//           The running maximum is only moved, and O rescaled in TMEM, when a block's maximum
//           exceeds it by more than 8 (log2 units), so probabilities stay below 2^8.
// At the end every row is divided by its sum and written as bf16. All waits are bounded.
// Key splits (gridDim.z = S > 1, the S CTAs of a row block forming a cluster along z): CTA s takes
// the key blocks [s nb / S, (s + 1) nb / S). Past its key loop each CTA writes its rows'
// unnormalised fp32 outputs and (m, l) to its slot of a workspace in global memory (row-fastest,
// so a warp's 16-byte stores are contiguous); after a cluster barrier (release / acquire at
// cluster scope) CTA s combines rows [s ceil(128 / S), ..) over the splits in split order,
// o = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s, and writes bf16. The exchange goes through
// L2 because the distributed shared memory takes a CTA's 128 rows at about 21 GB/s per SM.
// The LLM prefill runs the same kernel with no separate prefix (P = 0) and its prompt tokens as
// the S query tokens, every key visible (nctx = 0).

#pragma once

#include <cuda_bf16.h>
#include <cmath>

#include "ptx.h"

namespace jpi {
namespace {

constexpr int T5_ERR_LOAD = 1, T5_ERR_MMA = 2;
constexpr int T5_ROWS = 128;
constexpr int T5_KEYS = 64;
constexpr int T5_STAGES = 2;
constexpr int T5_THREADS = 256;
constexpr uint64_t T5_WAIT_NS = 200ull * 1000 * 1000;
constexpr float T5_RESCALE = 8.f;   // log2 units

struct T5Args {
    int S, H, P, kv_rows, maxB, layer;
    int nctx;           // suffix rows 0..nctx-1 (state, context tokens) see P + nctx keys
    float scale_log2;   // log2(e) / sqrt(D)
    __nv_bfloat16* o;   // [Mt][H][D]
    int* err;
    // Key splits: [CTA][D / 4][128] partial outputs and [CTA][128] (m, l), CTA = (row block,
    // request, split) in launch order; unused (null) without splits.
    float4* ws = nullptr;
    float2* wml = nullptr;
};

template <int D>
struct T5Smem {
    static constexpr int QBYTES = T5_ROWS * D * 2;        // D/64 blocks of [128 rows][128 B]
    static constexpr int KVBYTES = T5_KEYS * D * 2;       // D/64 blocks of [64 rows][128 B]
    static constexpr int STAGE = 2 * KVBYTES;             // ring slot s: K then V
    static constexpr int ST_OFF = QBYTES;
    static constexpr int PBYTES = T5_ROWS * T5_KEYS * 2;      // one P buffer [128 rows][128 B]
    static constexpr int P_OFF = ST_OFF + T5_STAGES * STAGE;   // two P buffers
    static constexpr int BAR_OFF = P_OFF + 2 * PBYTES;
    static constexpr int TOTAL = BAR_OFF + 256;
    static constexpr int TMEM_COLS = D == 256 ? 512 : 256;   // 2 score buffers of 64 + O (D)
};

__device__ __forceinline__ uint32_t pack_bf16x2_t5(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}
// 2^x by the hardware approximation (PTX ex2.approx.ftz.f32, relative error ~2^-22).
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Combine of S key splits for rows [r_lo, r_lo + nown) of a row block whose split 0 has workspace
// slot `cta`: each row's weights 2^(m_s - M) / sum_s 2^(m_s - M) l_s into `wsm`, then items
// (16-byte chunk c, owned row rr), rows fastest, summed over the splits in split order. A thread
// fetches the partials of IB items for all splits before it combines and stores any of them:
// with a store between them, the next item's loads would wait for it (the compiler cannot tell
// the workspace from the output), one L2 round trip per item.
template <int D, int S>
__device__ __forceinline__ void t5_combine(const T5Args& a, size_t cta, int r_lo, int nown, float* wsm, int row0,
                                           int nrows, int b, bool ok_all, int tid) {
    if (tid < nown) {
        float2 ml[S];
#pragma unroll
        for (int sp = 0; sp < S; ++sp) ml[sp] = __ldcg(&a.wml[(cta + sp) * T5_ROWS + r_lo + tid]);
        float M = -INFINITY;
#pragma unroll
        for (int sp = 0; sp < S; ++sp) M = fmaxf(M, ml[sp].x);
        float w[S], lsum = 0.f;
#pragma unroll
        for (int sp = 0; sp < S; ++sp) {
            w[sp] = ml[sp].x == -INFINITY ? 0.f : ex2(ml[sp].x - M);
            lsum += w[sp] * ml[sp].y;
        }
        const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
#pragma unroll
        for (int sp = 0; sp < S; ++sp) wsm[tid * S + sp] = w[sp] * inv;
    }
    __syncthreads();
    constexpr int IB = 32 / S;
    const int nitems = nown * (D / 4);
    for (int base = tid; base < nitems; base += IB * T5_THREADS) {
        float4 v[IB][S];
#pragma unroll
        for (int i = 0; i < IB; ++i) {
            const int idx = base + i * T5_THREADS;
            if (idx < nitems) {
                const int c = idx / nown, rr = idx - c * nown;
#pragma unroll
                for (int sp = 0; sp < S; ++sp)
                    v[i][sp] = __ldcg(&a.ws[((cta + sp) * (size_t)(D / 4) + c) * T5_ROWS + r_lo + rr]);
            }
        }
#pragma unroll
        for (int i = 0; i < IB; ++i) {
            const int idx = base + i * T5_THREADS;
            if (idx < nitems) {
                const int c = idx / nown, rr = idx - c * nown;
                const int R = row0 + r_lo + rr;
                float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int sp = 0; sp < S; ++sp) {
                    const float w = wsm[rr * S + sp];
                    acc.x = fmaf(w, v[i][sp].x, acc.x);
                    acc.y = fmaf(w, v[i][sp].y, acc.y);
                    acc.z = fmaf(w, v[i][sp].z, acc.z);
                    acc.w = fmaf(w, v[i][sp].w, acc.w);
                }
                if (R < nrows && ok_all)
                    *(uint2*)(a.o + ((size_t)b * nrows + R) * D + c * 4) =
                        make_uint2(pack_bf16x2_t5(acc.x, acc.y), pack_bf16x2_t5(acc.z, acc.w));
            }
        }
    }
}

// The same combine for S = 2 or 4, where rows [r_lo, r_lo + 128 / S) are exactly the rows of
// 4 / S softmax warps: those warps left this CTA's own partial rows in shared memory (`own`,
// [chunk][row], and `own_ml`), and every combine thread keeps one row (tid mod 128 / S) for all its
// chunks, so it fetches that row's (m, l) of every split together with the partials (one L2 round
// trip, no block barrier) and forms the weights itself.
template <int D, int S>
__device__ __forceinline__ void t5_combine_rows(const T5Args& a, size_t cta, int split, const float4* own,
                                                const float2* own_ml, int row0, int nrows, int b, bool ok_all,
                                                int tid) {
    constexpr int NOWN = T5_ROWS / S;          // rows per split: 64 or 32
    constexpr int CSTEP = T5_THREADS / NOWN;   // chunks one pass of the block covers
    constexpr int NI = (D / 4) / CSTEP;        // chunks per thread
    static_assert(T5_THREADS % NOWN == 0 && (D / 4) % CSTEP == 0, "rows and chunks tile the block");
    const int rr = tid % NOWN, cb = tid / NOWN, r_lo = split * NOWN;
    float2 ml[S];
    float4 v[NI][S];
#pragma unroll
    for (int sp = 0; sp < S; ++sp) {
        if (sp == split) {
            ml[sp] = own_ml[rr];
        } else {
            ml[sp] = __ldcg(&a.wml[(cta + sp) * T5_ROWS + r_lo + rr]);
        }
    }
#pragma unroll
    for (int i = 0; i < NI; ++i) {
        const int c = cb + i * CSTEP;
#pragma unroll
        for (int sp = 0; sp < S; ++sp) {
            if (sp == split) v[i][sp] = own[c * NOWN + rr];
            else v[i][sp] = __ldcg(&a.ws[((cta + sp) * (size_t)(D / 4) + c) * T5_ROWS + r_lo + rr]);
        }
    }
    float M = -INFINITY;
#pragma unroll
    for (int sp = 0; sp < S; ++sp) M = fmaxf(M, ml[sp].x);
    float w[S], lsum = 0.f;
#pragma unroll
    for (int sp = 0; sp < S; ++sp) {
        w[sp] = ml[sp].x == -INFINITY ? 0.f : ex2(ml[sp].x - M);
        lsum += w[sp] * ml[sp].y;
    }
    const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
#pragma unroll
    for (int sp = 0; sp < S; ++sp) w[sp] *= inv;
    const int R = row0 + r_lo + rr;
    if (R >= nrows || !ok_all) return;
    __nv_bfloat16* orow = a.o + ((size_t)b * nrows + R) * D;
#pragma unroll
    for (int i = 0; i < NI; ++i) {
        const int c = cb + i * CSTEP;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int sp = 0; sp < S; ++sp) {
            acc.x = fmaf(w[sp], v[i][sp].x, acc.x);
            acc.y = fmaf(w[sp], v[i][sp].y, acc.y);
            acc.z = fmaf(w[sp], v[i][sp].z, acc.z);
            acc.w = fmaf(w[sp], v[i][sp].w, acc.w);
        }
        *(uint2*)(orow + c * 4) = make_uint2(pack_bf16x2_t5(acc.x, acc.y), pack_bf16x2_t5(acc.z, acc.w));
    }
}

template <int D>
__global__ void __launch_bounds__(T5_THREADS, 1) k_attn_t5(const __grid_constant__ CUtensorMap qmap,
                                                           const __grid_constant__ CUtensorMap kmap,
                                                           const __grid_constant__ CUtensorMap vmap,
                                                           const __grid_constant__ T5Args a) {
    using L = T5Smem<D>;
    constexpr int NDB = D / 64;   // 64-column blocks of a row
    constexpr uint32_t IDESC_S = ptx::idesc_bf16_f32(T5_ROWS, T5_KEYS);
    constexpr uint32_t IDESC_PV = ptx::idesc_bf16_f32(T5_ROWS, D) | (1u << 16);   // B MN-major
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (ptx::smem_u32(smem_raw) & 1023u)) & 1023u);
    uint8_t* qs = smem;
    uint8_t* stages = smem + L::ST_OFF;
    uint8_t* ps = smem + L::P_OFF;
    uint64_t* bars = (uint64_t*)(smem + L::BAR_OFF);
    uint64_t* qfull = bars;                       // 1
    uint64_t* sfull = bars + 1;                   // 2: score buffer b ready
    uint64_t* pfull = bars + 3;                   // 2: P buffer b written by the 128 softmax threads
    uint64_t* odone = bars + 5;                   // 2: P V of the block in P buffer b done
    // K and V have their own rings (slot i mod 2), so K of block i+2 is fetched as soon as
    // S_i is done and V of block i+2 once P_i V_i is done.
    uint64_t* kfull = bars + 7;                   // T5_STAGES
    uint64_t* vfull = kfull + T5_STAGES;
    uint64_t* kempty = vfull + T5_STAGES;
    uint64_t* vempty = kempty + T5_STAGES;
    uint32_t* tmem_slot = (uint32_t*)(vempty + T5_STAGES);
    int* flag = (int*)(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int rb = blockIdx.x, b = blockIdx.y;
    const int nrows = a.S * a.H, nk = a.P + a.S;
    const int row0 = rb * T5_ROWS;
    // Key split: this CTA's key blocks blk0 .. blk0 + nb - 1 of the request's nb_all.
    const int nsplit = (int)gridDim.z, split = (int)blockIdx.z;
    const int nb_all = (nk + T5_KEYS - 1) / T5_KEYS;
    const int blk0 = split * nb_all / nsplit;
    const int nb = (split + 1) * nb_all / nsplit - blk0;
    float x_m = -INFINITY, x_l = 0.f;   // the row's running maximum and sum (softmax threads)

    if (warp == 1) {
        ptx::tmem_alloc(tmem_slot, L::TMEM_COLS);
        ptx::tmem_relinquish();
    }
    if (tid == 0) {
        ptx::mbar_init(qfull, 1);
        ptx::mbar_init(&sfull[0], 1);
        ptx::mbar_init(&sfull[1], 1);
        for (int b2 = 0; b2 < 2; ++b2) {
            ptx::mbar_init(&pfull[b2], 128);
            ptx::mbar_init(&odone[b2], 1);
        }
        for (int s = 0; s < T5_STAGES; ++s) {
            ptx::mbar_init(&kfull[s], 1);
            ptx::mbar_init(&vfull[s], 1);
            ptx::mbar_init(&kempty[s], 1);
            ptx::mbar_init(&vempty[s], 1);
        }
        ptx::fence_mbar_init();
        *flag = 0;
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp <= 1) {
        // Warp 0 streams Q and K, warp 1 streams V.
        if (lane == 0) {
            const bool is_v = warp == 1;
            const uint64_t pol = ptx::l2_policy_evict_first();
            const int kv0 = (a.layer * a.maxB + b) * a.kv_rows;
            uint64_t* fullb = is_v ? vfull : kfull;
            uint64_t* emptyb = is_v ? vempty : kempty;
            const CUtensorMap* map = is_v ? &vmap : &kmap;
            // Block i into ring slot i mod 2: NDB column boxes.
            auto load = [&](int i) {
                const int sl = i % T5_STAGES;
                uint8_t* base = stages + sl * L::STAGE + (is_v ? L::KVBYTES : 0);
                ptx::mbar_expect_tx(&fullb[sl], (uint32_t)L::KVBYTES);
                for (int db = 0; db < NDB; ++db)
                    ptx::tma_load_2d(base + db * (T5_KEYS * 128), map, &fullb[sl], db * 64,
                                     kv0 + (blk0 + i) * T5_KEYS, pol);
            };
            // First use of both slots: blocks made only of prefix keys were written before this
            // graph ran and are fetched before the dependency wait.
            int first = 0;
            while (first < T5_STAGES && first < nb && (blk0 + first + 1) * T5_KEYS <= a.P) load(first++);
            if (!is_v) ptx::prefetch_tmap(&qmap);
            ptx::grid_dep_wait();
            if (!is_v) {
                ptx::mbar_expect_tx(qfull, (uint32_t)L::QBYTES);
                for (int db = 0; db < NDB; ++db)
                    ptx::tma_load_2d(qs + db * (T5_ROWS * 128), &qmap, qfull, db * 64, b * nrows + row0, pol);
            }
            for (; first < T5_STAGES && first < nb; ++first) load(first);
            // Block j once the MMAs that read block j - 2 (S_{j-2}, or P_{j-2} V_{j-2}) are done.
            for (int j = T5_STAGES; j < nb; ++j) {
                if (!ptx::mbar_wait_bounded(&emptyb[j % T5_STAGES], ((j - 2) >> 1) & 1, T5_WAIT_NS)) {
                    *flag = T5_ERR_LOAD;
                    break;
                }
                load(j);
            }
        }
    } else if (warp == 2) {
        if (lane == 0) {
            const uint32_t qb = ptx::smem_u32(qs), sb = ptx::smem_u32(stages);
            bool good = ptx::mbar_wait_bounded(qfull, 0, T5_WAIT_NS);
            // S_i = Q K_i^T into score buffer i mod 2; K slot i mod 2 is released when it is done.
            auto issue_s = [&](int i) {
                const int sl = i % T5_STAGES;
                if (!ptx::mbar_wait_bounded(&kfull[sl], (i >> 1) & 1, T5_WAIT_NS)) good = false;
                ptx::tc_fence_after();
                if (good) {
                    const uint32_t kb = sb + sl * L::STAGE;
                    for (int db = 0; db < NDB; ++db)
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            ptx::mma_bf16(tmem + (uint32_t)(64 * (i & 1)),
                                          ptx::desc_sw128(qb + db * (T5_ROWS * 128) + kk * 32),
                                          ptx::desc_sw128(kb + db * (T5_KEYS * 128) + kk * 32), IDESC_S,
                                          (db | kk) != 0);
                }
                ptx::mma_commit(&sfull[i & 1]);
                if (i + T5_STAGES < nb) ptx::mma_commit(&kempty[sl]);
            };
            if (nb > 0) issue_s(0);
            if (nb > 1) issue_s(1);
            // S_{i+2} once P_i is written: the softmax of block i has read score buffer i mod 2.
            for (int i = 0; i + 2 < nb; ++i) {
                if (!ptx::mbar_wait_bounded(&pfull[i & 1], (i >> 1) & 1, T5_WAIT_NS)) good = false;
                ptx::tc_fence_after();
                issue_s(i + 2);
            }
            if (!good) *flag = T5_ERR_MMA;
        }
    } else if (warp == 3) {
        if (lane == 0) {
            const uint32_t sb = ptx::smem_u32(stages), pb = ptx::smem_u32(ps);
            bool good = true;
            for (int i = 0; i < nb; ++i) {
                const int sl = i % T5_STAGES;
                if (!ptx::mbar_wait_bounded(&pfull[i & 1], (i >> 1) & 1, T5_WAIT_NS)) good = false;
                if (!ptx::mbar_wait_bounded(&vfull[sl], (i >> 1) & 1, T5_WAIT_NS)) good = false;
                ptx::tc_fence_after();
                if (good) {
                    const uint32_t vb = sb + sl * L::STAGE + L::KVBYTES;
                    const uint32_t pbi = pb + (uint32_t)((i & 1) * L::PBYTES);
#pragma unroll
                    for (int kk = 0; kk < T5_KEYS / 16; ++kk)
                        ptx::mma_bf16(tmem + 128u, ptx::desc_sw128(pbi + kk * 32),
                                      ptx::desc_sw128_mn(vb + kk * 16 * 128, T5_KEYS * 128, 1024), IDESC_PV,
                                      (i | kk) != 0);
                }
                if (i + T5_STAGES < nb) ptx::mma_commit(&vempty[sl]);
                ptx::mma_commit(&odone[i & 1]);
            }
            if (!good) *flag = T5_ERR_MMA;
        }
    } else {
        // ---- softmax: one query row per thread ----
        const int row = (warp & 3) * 32 + lane;
        const int R = row0 + row;
        const bool valid = R < nrows;
        // Visible keys: state and context rows see the prefix and each other; padding rows none.
        const int nvis = !valid ? 0 : R / a.H < a.nctx ? a.P + a.nctx : nk;
        const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
        float m_used = -INFINITY, l = 0.f;
        bool good = true;
        for (int i = 0; i < nb; ++i) {
            if (!ptx::mbar_wait_bounded(&sfull[i & 1], (i >> 1) & 1, T5_WAIT_NS)) good = false;
            ptx::tc_fence_after();
            // The block's 64 raw scores: four loads in flight, one wait.
            uint32_t r[4][16];
            {
                const uint32_t sa = lane_base + (uint32_t)(64 * (i & 1));
                ptx::tmem_ld_x16(sa, r[0]);
                ptx::tmem_ld_x16(sa + 16u, r[1]);
                ptx::tmem_ld_x16(sa + 32u, r[2]);
                ptx::tmem_ld_x16(sa + 48u, r[3]);
                ptx::tmem_ld_wait();
            }
            // Keys of this block the row sees: all of them except in the last block(s).
            const int vis = nvis - (blk0 + i) * T5_KEYS;
            const bool full = vis >= T5_KEYS;
            // Block maximum in log2 units (the scale is positive, so it commutes with the max);
            // four independent chains.
            float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
            for (int j = 0; j < 16; ++j)
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    if (full || 16 * q + j < vis) m4[q] = fmaxf(m4[q], __uint_as_float(r[q][j]));
            const float mb = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3])) * a.scale_log2;
            const bool move = mb > m_used + T5_RESCALE;
            const float alpha = !move ? 1.f : m_used == -INFINITY ? 0.f : ex2(m_used - mb);
            // TMEM loads and stores are warp-collective: the warp rescales together, lanes whose
            // maximum stays put multiply by 1. O is settled once P V of the previous block is done.
            if (__any_sync(0xffffffffu, move && i > 0 && m_used != -INFINITY)) {
                if (!ptx::mbar_wait_bounded(&odone[(i - 1) & 1], ((i - 1) >> 1) & 1, T5_WAIT_NS)) good = false;
                ptx::tc_fence_after();
#pragma unroll 1
                for (int c0 = 0; c0 < D; c0 += 16) {
                    uint32_t ro[16];
                    ptx::tmem_ld_x16(lane_base + 128u + (uint32_t)c0, ro);
                    ptx::tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < 16; ++j) ro[j] = __float_as_uint(__uint_as_float(ro[j]) * alpha);
                    ptx::tmem_st_x16(lane_base + 128u + (uint32_t)c0, ro);
                }
                ptx::tmem_st_wait();
            }
            if (move) {
                l *= alpha;
                m_used = mb;
            }
            // p = 2^(s * scale - m): one FMA and one exp per key; zero for hidden keys and while
            // the row has seen no key at all. Four partial sums.
            const bool seen = m_used != -INFINITY;
            const float neg_m = seen ? -m_used : 0.f;
            float l4[4] = {0.f, 0.f, 0.f, 0.f};
            uint32_t pk[T5_KEYS / 2];
#pragma unroll
            for (int q = 0; q < 4; ++q)
#pragma unroll
                for (int j = 0; j < 16; j += 2) {
                    const int k = 16 * q + j;
                    float p0 = ex2(fmaf(__uint_as_float(r[q][j]), a.scale_log2, neg_m));
                    float p1 = ex2(fmaf(__uint_as_float(r[q][j + 1]), a.scale_log2, neg_m));
                    if (!full || !seen) {
                        p0 = (seen && k < vis) ? p0 : 0.f;
                        p1 = (seen && k + 1 < vis) ? p1 : 0.f;
                    }
                    l4[q] += p0 + p1;
                    pk[k / 2] = pack_bf16x2_t5(p0, p1);
                }
            l += (l4[0] + l4[1]) + (l4[2] + l4[3]);
            // P buffer i mod 2 is free once P V of block i - 2 is done.
            if (i >= 2 && !ptx::mbar_wait_bounded(&odone[i & 1], ((i - 2) >> 1) & 1, T5_WAIT_NS)) good = false;
            ptx::tc_fence_after();
            // Row `row` of P: 8 chunks of 16 bytes, chunk c at position c ^ (row mod 8).
            uint4* prow = (uint4*)(ps + (i & 1) * L::PBYTES + row * 128);
#pragma unroll
            for (int c = 0; c < 8; ++c)
                prow[c ^ (row & 7)] = make_uint4(pk[4 * c], pk[4 * c + 1], pk[4 * c + 2], pk[4 * c + 3]);
            ptx::fence_proxy_async_smem();
            ptx::tc_fence_before();
            ptx::mbar_arrive(&pfull[i & 1]);
        }
        // Every P V is done (both buffers' last commits observed, so none arrives after exit).
        if (nb >= 2 && !ptx::mbar_wait_bounded(&odone[(nb - 2) & 1], ((nb - 2) >> 1) & 1, T5_WAIT_NS)) good = false;
        if (nb >= 1 && !ptx::mbar_wait_bounded(&odone[(nb - 1) & 1], ((nb - 1) >> 1) & 1, T5_WAIT_NS)) good = false;
        ptx::tc_fence_after();
        ptx::grid_dep_launch();
        if (!good) *flag = T5_ERR_MMA;
        x_m = m_used;
        x_l = l;
        const float inv = l > 0.f ? 1.f / l : 0.f;
        __nv_bfloat16* orow = a.o + ((size_t)b * nrows + R) * D;
#pragma unroll 1
        for (int c0 = 0; c0 < D && nsplit == 1; c0 += 32) {
            uint32_t r[2][16];
            ptx::tmem_ld_x16(lane_base + 128u + (uint32_t)c0, r[0]);
            ptx::tmem_ld_x16(lane_base + 128u + (uint32_t)(c0 + 16), r[1]);
            ptx::tmem_ld_wait();
            if (valid && good) {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    uint32_t w8[8];
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        w8[j] = pack_bf16x2_t5(__uint_as_float(r[h][2 * j]) * inv,
                                               __uint_as_float(r[h][2 * j + 1]) * inv);
                    uint4* dst = (uint4*)(orow + c0 + 16 * h);
                    dst[0] = make_uint4(w8[0], w8[1], w8[2], w8[3]);
                    dst[1] = make_uint4(w8[4], w8[5], w8[6], w8[7]);
                }
            }
        }
    }

    if (nsplit > 1) {
        // ---- combine the key splits of this row block through the workspace ----
        const size_t cta = ((size_t)blockIdx.y * gridDim.x + blockIdx.x) * nsplit;   // split 0 of the row block
        // With 2 or 4 splits the rows this CTA combines are whole warps' rows: those warps keep
        // their partials in shared memory (over the query tile; every MMA is done) and their
        // (m, l) over the P buffers.
        const bool rows_fixed = nsplit == 2 || nsplit == 4;
        const int nown_fixed = rows_fixed ? T5_ROWS / nsplit : 0;
        float4* own = reinterpret_cast<float4*>(smem);
        float2* own_ml = reinterpret_cast<float2*>(ps);
        if (warp >= 4) {
            const int row = (warp & 3) * 32 + lane;
            const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
            const bool mine = rows_fixed && row / nown_fixed == split;   // warp-uniform
            float4* dst = mine ? own + (row - split * nown_fixed) : a.ws + (cta + split) * (size_t)(D / 4) * T5_ROWS + row;
            const int stride = mine ? nown_fixed : T5_ROWS;
#pragma unroll 1
            for (int c0 = 0; c0 < D; c0 += 32) {
                uint32_t r[2][16];
                ptx::tmem_ld_x16(lane_base + 128u + (uint32_t)c0, r[0]);
                ptx::tmem_ld_x16(lane_base + 128u + (uint32_t)(c0 + 16), r[1]);
                ptx::tmem_ld_wait();
#pragma unroll
                for (int v = 0; v < 8; ++v)
                    dst[(size_t)(c0 / 4 + v) * stride] =
                        make_float4(__uint_as_float(r[v >> 2][4 * (v & 3)]), __uint_as_float(r[v >> 2][4 * (v & 3) + 1]),
                                    __uint_as_float(r[v >> 2][4 * (v & 3) + 2]), __uint_as_float(r[v >> 2][4 * (v & 3) + 3]));
            }
            if (mine) own_ml[row - split * nown_fixed] = make_float2(x_m, x_l);
            else a.wml[(cta + split) * T5_ROWS + row] = make_float2(x_m, x_l);
        }
        // Every split's rows are in the workspace (the barrier orders global memory at cluster scope;
        // the reads below go to L2, past this SM's L1).
        ptx::tc_fence_before();
        ptx::cluster_sync_all();
        ptx::tc_fence_after();
        float* wsm = reinterpret_cast<float*>(smem);   // [rows][S] weights, over the query tile
        const int rps = (T5_ROWS + nsplit - 1) / nsplit;
        const int r_lo = split * rps;
        const int nown = max(0, min(T5_ROWS, r_lo + rps) - r_lo);
        const bool ok_all = *flag == 0;   // written before the cluster barrier
        // The launcher splits 2, 3 or 4 ways.
        if (nsplit == 2) t5_combine_rows<D, 2>(a, cta, split, own, own_ml, row0, nrows, b, ok_all, tid);
        else if (nsplit == 4) t5_combine_rows<D, 4>(a, cta, split, own, own_ml, row0, nrows, b, ok_all, tid);
        else t5_combine<D, 3>(a, cta, r_lo, nown, wsm, row0, nrows, b, ok_all, tid);
    }

    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (tid == 0 && *flag != 0) atomicCAS(a.err, 0, *flag);
    if (warp == 1) ptx::tmem_dealloc(tmem, L::TMEM_COLS);
}

}  // namespace
}  // namespace jpi
