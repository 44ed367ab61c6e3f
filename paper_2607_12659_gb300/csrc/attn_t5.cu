// Suffix attention on tcgen05 tensor cores for batched launches, without key splits.
//
// App. A of the paper: the expert's queries (state token + C action tokens, all H heads) attend
// over the matching LLM layer's KV cache followed by the suffix's own keys/values; one KV head
// is shared by all heads, so one request is a dense [S*H] x [P+S] problem (rows token-major,
// row = i * H + head; the state row i = 0 sees the prefix and itself only).
//
// One CTA = 128 query rows of one request over all of its keys, in blocks of 64 keys:
//   warp 0  one thread: bulk tensor copies of the query tile once, then (K, V) blocks through a
//           two-stage ring (prefix blocks may be fetched before the grid-dependency wait);
//   warp 1  one thread: S_i = Q K_i^T (M = 128, N = 64, K = D) into one of two TMEM score
//           buffers, then O += P_i V_i (M = 128, N = D, K = 64) into the TMEM output with V read
//           as an MN-major operand straight from its bulk copy;
//   warps 2-5  one query row per thread (its TMEM lane): scale, mask, block maximum, softmax
//           probabilities P_i written to shared memory (bf16, 128-byte swizzled K-major rows).
//           The running maximum is only moved, and O rescaled in TMEM, when a block's maximum
//           exceeds it by more than 8 (log2 units), so probabilities stay below 2^8.
// At the end every row is divided by its sum and written as bf16. All waits are bounded.

#include "jpi_internal.h"
#include "ptx.h"
#include "tc_path.h"

#include <cmath>
#include <cstdlib>

namespace jpi {
namespace {

constexpr int T5_ROWS = 128;
constexpr int T5_KEYS = 64;
constexpr int T5_STAGES = 2;
constexpr int T5_THREADS = 192;
constexpr uint64_t T5_WAIT_NS = 200ull * 1000 * 1000;
constexpr float T5_RESCALE = 8.f;   // log2 units

struct T5Args {
    int S, H, P, kv_rows, maxB, layer;
    float scale_log2;   // log2(e) / sqrt(D)
    __nv_bfloat16* o;   // [Mt][H][D]
    int* err;
};

template <int D>
struct T5Smem {
    static constexpr int QBYTES = T5_ROWS * D * 2;        // D/64 blocks of [128 rows][128 B]
    static constexpr int KVBYTES = T5_KEYS * D * 2;       // D/64 blocks of [64 rows][128 B]
    static constexpr int STAGE = 2 * KVBYTES;             // K then V
    static constexpr int ST_OFF = QBYTES;
    static constexpr int P_OFF = ST_OFF + T5_STAGES * STAGE;
    static constexpr int BAR_OFF = P_OFF + T5_ROWS * T5_KEYS * 2;
    static constexpr int TOTAL = BAR_OFF + 128;
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
    uint64_t* pfull = bars + 3;                   // 1: P written by the 128 softmax threads
    uint64_t* odone = bars + 4;                   // 1: P V of the block done
    uint64_t* stfull = bars + 5;                  // T5_STAGES
    uint64_t* stempty = stfull + T5_STAGES;       // T5_STAGES
    uint32_t* tmem_slot = (uint32_t*)(stempty + T5_STAGES);
    int* flag = (int*)(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int rb = blockIdx.x, b = blockIdx.y;
    const int nrows = a.S * a.H, nk = a.P + a.S;
    const int row0 = rb * T5_ROWS;
    const int nb = (nk + T5_KEYS - 1) / T5_KEYS;

    if (warp == 1) {
        ptx::tmem_alloc(tmem_slot, L::TMEM_COLS);
        ptx::tmem_relinquish();
    }
    if (tid == 0) {
        ptx::mbar_init(qfull, 1);
        ptx::mbar_init(&sfull[0], 1);
        ptx::mbar_init(&sfull[1], 1);
        ptx::mbar_init(pfull, 128);
        ptx::mbar_init(odone, 1);
        for (int s = 0; s < T5_STAGES; ++s) {
            ptx::mbar_init(&stfull[s], 1);
            ptx::mbar_init(&stempty[s], 1);
        }
        ptx::fence_mbar_init();
        *flag = 0;
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            const uint64_t pol = ptx::l2_policy_evict_first();
            const int kv0 = (a.layer * a.maxB + b) * a.kv_rows;
            auto load_kv = [&](int i, int s) {
                uint8_t* st = stages + s * L::STAGE;
                ptx::mbar_expect_tx(&stfull[s], (uint32_t)L::STAGE);
                for (int db = 0; db < NDB; ++db) {
                    ptx::tma_load_2d(st + db * (T5_KEYS * 128), &kmap, &stfull[s], db * 64, kv0 + i * T5_KEYS, pol);
                    ptx::tma_load_2d(st + L::KVBYTES + db * (T5_KEYS * 128), &vmap, &stfull[s], db * 64,
                                     kv0 + i * T5_KEYS, pol);
                }
            };
            // Blocks made only of prefix keys were written before this graph ran.
            int pre = 0;
            while (pre < T5_STAGES && pre < nb && (pre + 1) * T5_KEYS <= a.P) {
                load_kv(pre, pre);
                ++pre;
            }
            ptx::prefetch_tmap(&qmap);
            ptx::grid_dep_wait();
            ptx::mbar_expect_tx(qfull, (uint32_t)L::QBYTES);
            for (int db = 0; db < NDB; ++db)
                ptx::tma_load_2d(qs + db * (T5_ROWS * 128), &qmap, qfull, db * 64, b * nrows + row0, pol);
            for (int i = pre; i < nb; ++i) {
                const int s = i % T5_STAGES, n = i / T5_STAGES;
                if (i >= T5_STAGES && !ptx::mbar_wait_bounded(&stempty[s], (n - 1) & 1, T5_WAIT_NS)) {
                    *flag = DEV_TIMEOUT_WEIGHTS;
                    break;
                }
                load_kv(i, s);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t qb = ptx::smem_u32(qs), sb = ptx::smem_u32(stages), pb = ptx::smem_u32(ps);
            bool good = ptx::mbar_wait_bounded(qfull, 0, T5_WAIT_NS);
            auto issue_s = [&](int i) {
                const int s = i % T5_STAGES;
                if (!ptx::mbar_wait_bounded(&stfull[s], (i / T5_STAGES) & 1, T5_WAIT_NS)) good = false;
                ptx::tc_fence_after();
                if (good) {
                    const uint32_t kb = sb + s * L::STAGE;
                    for (int db = 0; db < NDB; ++db)
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            ptx::mma_bf16(tmem + (uint32_t)(64 * (i & 1)),
                                          ptx::desc_sw128(qb + db * (T5_ROWS * 128) + kk * 32),
                                          ptx::desc_sw128(kb + db * (T5_KEYS * 128) + kk * 32), IDESC_S,
                                          (db | kk) != 0);
                }
                ptx::mma_commit(&sfull[i & 1]);
            };
            issue_s(0);
            for (int i = 0; i < nb; ++i) {
                if (i + 1 < nb) issue_s(i + 1);
                if (!ptx::mbar_wait_bounded(pfull, i & 1, T5_WAIT_NS)) good = false;
                ptx::tc_fence_after();
                if (good) {
                    const uint32_t vb = sb + (i % T5_STAGES) * L::STAGE + L::KVBYTES;
#pragma unroll
                    for (int kk = 0; kk < T5_KEYS / 16; ++kk)
                        ptx::mma_bf16(tmem + 128u, ptx::desc_sw128(pb + kk * 32),
                                      ptx::desc_sw128_mn(vb + kk * 16 * 128, T5_KEYS * 128, 1024), IDESC_PV,
                                      (i | kk) != 0);
                }
                if (i + T5_STAGES < nb) ptx::mma_commit(&stempty[i % T5_STAGES]);
                ptx::mma_commit(odone);
            }
            if (!good) *flag = DEV_TIMEOUT_MMA;
        }
    } else {
        // ---- softmax: one query row per thread ----
        const int row = (warp & 3) * 32 + lane;
        const int R = row0 + row;
        const bool valid = R < nrows;
        // Visible keys: the state row sees the prefix and itself; padding rows see none.
        const int nvis = !valid ? 0 : R / a.H == 0 ? a.P + 1 : nk;
        const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
        float m_used = -INFINITY, l = 0.f;
        bool good = true;
        for (int i = 0; i < nb; ++i) {
            if (!ptx::mbar_wait_bounded(&sfull[i & 1], (i >> 1) & 1, T5_WAIT_NS)) good = false;
            ptx::tc_fence_after();
            float s[T5_KEYS];
#pragma unroll
            for (int c0 = 0; c0 < T5_KEYS; c0 += 16) {
                uint32_t r[16];
                ptx::tmem_ld_x16(lane_base + (uint32_t)(64 * (i & 1) + c0), r);
                ptx::tmem_ld_wait();
#pragma unroll
                for (int j = 0; j < 16; ++j) s[c0 + j] = __uint_as_float(r[j]);
            }
            const int key0 = i * T5_KEYS;
            float mb = -INFINITY;
#pragma unroll
            for (int j = 0; j < T5_KEYS; ++j) {
                s[j] = key0 + j < nvis ? s[j] * a.scale_log2 : -INFINITY;
                mb = fmaxf(mb, s[j]);
            }
            // P V of the previous block is done: the P buffer is free and O is settled.
            if (i > 0 && !ptx::mbar_wait_bounded(odone, (i - 1) & 1, T5_WAIT_NS)) good = false;
            ptx::tc_fence_after();
            const bool move = mb > m_used + T5_RESCALE;
            const float alpha = !move ? 1.f : m_used == -INFINITY ? 0.f : ex2(m_used - mb);
            // TMEM loads and stores are warp-collective: the warp rescales together, lanes whose
            // maximum stays put multiply by 1.
            if (__any_sync(0xffffffffu, move && i > 0 && m_used != -INFINITY)) {
#pragma unroll 1
                for (int c0 = 0; c0 < D; c0 += 16) {
                    uint32_t r[16];
                    ptx::tmem_ld_x16(lane_base + 128u + (uint32_t)c0, r);
                    ptx::tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < 16; ++j) r[j] = __float_as_uint(__uint_as_float(r[j]) * alpha);
                    ptx::tmem_st_x16(lane_base + 128u + (uint32_t)c0, r);
                }
                ptx::tmem_st_wait();
            }
            if (move) {
                l *= alpha;
                m_used = mb;
            }
            uint32_t pk[T5_KEYS / 2];
#pragma unroll
            for (int j = 0; j < T5_KEYS; j += 2) {
                const float p0 = s[j] == -INFINITY ? 0.f : ex2(s[j] - m_used);
                const float p1 = s[j + 1] == -INFINITY ? 0.f : ex2(s[j + 1] - m_used);
                l += p0 + p1;
                pk[j / 2] = pack_bf16x2_t5(p0, p1);
            }
            // Row `row` of P: 8 chunks of 16 bytes, chunk c at position c ^ (row mod 8).
            uint4* prow = (uint4*)(ps + row * 128);
#pragma unroll
            for (int c = 0; c < 8; ++c)
                prow[c ^ (row & 7)] = make_uint4(pk[4 * c], pk[4 * c + 1], pk[4 * c + 2], pk[4 * c + 3]);
            ptx::fence_proxy_async_smem();
            ptx::tc_fence_before();
            ptx::mbar_arrive(pfull);
        }
        if (!ptx::mbar_wait_bounded(odone, (nb - 1) & 1, T5_WAIT_NS)) good = false;
        ptx::tc_fence_after();
        ptx::grid_dep_launch();
        if (!good) *flag = DEV_TIMEOUT_MMA;
        const float inv = l > 0.f ? 1.f / l : 0.f;
        __nv_bfloat16* orow = a.o + ((size_t)b * nrows + R) * D;
#pragma unroll 1
        for (int c0 = 0; c0 < D; c0 += 16) {
            uint32_t r[16];
            ptx::tmem_ld_x16(lane_base + 128u + (uint32_t)c0, r);
            ptx::tmem_ld_wait();
            if (valid && good) {
                uint32_t w8[8];
#pragma unroll
                for (int j = 0; j < 8; ++j)
                    w8[j] = pack_bf16x2_t5(__uint_as_float(r[2 * j]) * inv, __uint_as_float(r[2 * j + 1]) * inv);
                uint4* dst = (uint4*)(orow + c0);
                dst[0] = make_uint4(w8[0], w8[1], w8[2], w8[3]);
                dst[1] = make_uint4(w8[4], w8[5], w8[6], w8[7]);
            }
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (tid == 0 && *flag != 0) atomicCAS(a.err, 0, *flag);
    if (warp == 1) ptx::tmem_dealloc(tmem, L::TMEM_COLS);
}

template <int D>
jpi_status prepare_t5(jpi_handle* h) {
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_attn_t5<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      1024 + T5Smem<D>::TOTAL));
    return JPI_OK;
}

template <int D>
jpi_status launch_t5(jpi_handle* h, int l, int B, int C, cudaStream_t st) {
    T5Args a;
    a.S = C + 1;
    a.H = h->H;
    a.P = h->cur_prefix;
    a.kv_rows = h->kv_rows;
    a.maxB = h->maxB;
    a.layer = l;
    a.scale_log2 = 1.4426950408889634f / sqrtf((float)D);
    a.o = (__nv_bfloat16*)h->o;
    a.err = h->dev_err;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((a.S * a.H + T5_ROWS - 1) / T5_ROWS, B);
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
    h->attn_t5_min_batch = env ? std::atoi(env) : 8;
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
