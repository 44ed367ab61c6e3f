// Time conditioning's largest product on tensor cores: the adaptive-norm modulation vectors of
// every layer for all N step times at once (App. A, Tab. arch: the expert's adaRMSNorm scales,
// shifts and gates are functions of the flow time only, so one pass over the stacked matrix
// serves the whole denoise).
//
//   Y[n][r] = sum_k M[r][k] X[n][k] + b[r],   r < R = (6 L + 2) W,  k < W,  n < N <= 16.
//
// M (bf16, [R][W] row-major, 230.7 MB at pi0.5 sizes) is streamed from HBM exactly once by bulk
// tensor copies (128-row x 64-column boxes, 128-byte swizzle) and is the A operand (M = 128) of
// tcgen05.mma. The B operand is X split into two bf16 parts, hi = bf16(x) and lo = bf16(x - hi),
// stacked as rows 0..15 (hi) and 16..31 (lo) of a 32-row operand kept in shared memory for the
// whole kernel, so the fp32 inputs enter with about 16 significant bits: D[r][n] + D[r][16 + n]
// is the product to within 2^-17 of |M||X| per term, accumulated in fp32 (TMEM).
//
// Persistent: one CTA per SM walks the 128-row tiles t = blockIdx.x, + gridDim.x, ...
//   warp 0  one thread streams the tile's 64-column weight blocks into a ring of stages;
//   warp 1  one thread issues 4 MMAs (M = 128, N = 32, K = 16) per block into one of two TMEM
//           accumulators (32 columns each) and frees each stage through tcgen05.commit;
//   warps 4-7  read a finished accumulator (one weight row per thread), add the two halves and
//           the bias, and store the N outputs of that row (consecutive rows in consecutive lanes).
// The first stages of weights are requested before the dependency wait on the kernel that
// produced X. Every wait is bounded; on a timeout the kernel records a device error and returns.

#include "tc_path.h"
#include "ptx.h"

namespace jpi {
namespace {

constexpr int MT_ROWS = 128;
constexpr int MT_KBLK = 64;
constexpr int MT_N = 32;                       // MMA N: 16 hi rows + 16 lo rows
constexpr int MT_STAGES = 8;
constexpr int MT_THREADS = 256;
constexpr int MT_WBYTES = MT_ROWS * MT_KBLK * 2;   // 16 KB weight block
constexpr int MT_XBLK = MT_N * MT_KBLK * 2;       // 4 KB operand block
constexpr uint64_t MT_WAIT_NS = 200ull * 1000 * 1000;

__host__ __device__ constexpr size_t mod_tc_smem(int K) {
    // operand blocks | weight ring | barriers (full, empty, acc full[2], acc empty[2]) + TMEM slot + flag
    return (size_t)(K / MT_KBLK) * MT_XBLK + (size_t)MT_STAGES * MT_WBYTES + 256;
}

__device__ __forceinline__ uint32_t bf16_bits(__nv_bfloat16 v) {
    return (uint32_t)*reinterpret_cast<unsigned short*>(&v);
}

__global__ void __launch_bounds__(MT_THREADS, 1) k_mod_tc(const __grid_constant__ CUtensorMap wmap,
                                                        const float* __restrict__ X,
                                                        const float* __restrict__ bias,
                                                        float* __restrict__ Y, int N, int R, int K,
                                                        int* err) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (ptx::smem_u32(smem_raw) & 1023u)) & 1023u);
    const int nkb = K / MT_KBLK;
    uint8_t* xop = smem;                                  // [nkb][32 rows][128 B], swizzled
    uint8_t* ring = smem + (size_t)nkb * MT_XBLK;         // [STAGES][16 KB]
    uint64_t* full = (uint64_t*)(ring + (size_t)MT_STAGES * MT_WBYTES);
    uint64_t* empty = full + MT_STAGES;
    uint64_t* accf = empty + MT_STAGES;
    uint64_t* acce = accf + 2;
    uint32_t* tmem_slot = (uint32_t*)(acce + 2);
    int* flag = (int*)(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int ntiles = R / MT_ROWS;
    const int t0 = blockIdx.x, dt = gridDim.x;
    const int my_tiles = t0 < ntiles ? (ntiles - t0 + dt - 1) / dt : 0;
    const int total = my_tiles * nkb;   // weight blocks this CTA streams

    if (warp == 1) {
        ptx::tmem_alloc(tmem_slot, 2 * MT_N);
        ptx::tmem_relinquish();
    }
    if (tid == 0) {
        for (int i = 0; i < 2 * MT_STAGES; ++i) ptx::mbar_init(&full[i], 1);
        ptx::mbar_init(&accf[0], 1);
        ptx::mbar_init(&accf[1], 1);
        ptx::mbar_init(&acce[0], 128);
        ptx::mbar_init(&acce[1], 128);
        ptx::fence_mbar_init();
        *flag = 0;
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    const uint64_t pol = ptx::l2_policy_evict_first();
    auto load = [&](int it) {
        const int s = it % MT_STAGES;
        const int tile = t0 + (it / nkb) * dt, kb = it % nkb;
        ptx::mbar_expect_tx(&full[s], (uint32_t)MT_WBYTES);
        ptx::tma_load_2d(ring + (size_t)s * MT_WBYTES, &wmap, &full[s], kb * MT_KBLK, tile * MT_ROWS, pol);
    };
    // The weights do not depend on the previous kernel: fill the ring before waiting for it.
    const int npre = total < MT_STAGES ? total : MT_STAGES;
    if (tid == 0)
        for (int it = 0; it < npre; ++it) load(it);
    ptx::grid_dep_wait();

    // B operand: row n = hi(X[n]), row 16 + n = lo(X[n]) (zero for n >= N); 16-byte chunk c of a
    // 128-byte row sits at chunk c ^ (row mod 8) (the 128-byte swizzle the MMA descriptor names).
    for (int item = tid; item < 16 * (K / 8); item += MT_THREADS) {
        const int n = item / (K / 8), k0 = (item % (K / 8)) * 8;
        uint32_t hi[4] = {0u, 0u, 0u, 0u}, lo[4] = {0u, 0u, 0u, 0u};
        if (n < N) {
            const float4 a = *(const float4*)(X + (size_t)n * K + k0);
            const float4 b = *(const float4*)(X + (size_t)n * K + k0 + 4);
            const float v[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
            for (int e = 0; e < 8; e += 2) {
                const __nv_bfloat16 h0 = __float2bfloat16_rn(v[e]), h1 = __float2bfloat16_rn(v[e + 1]);
                const __nv_bfloat16 l0 = __float2bfloat16_rn(v[e] - __bfloat162float(h0));
                const __nv_bfloat16 l1 = __float2bfloat16_rn(v[e + 1] - __bfloat162float(h1));
                hi[e / 2] = bf16_bits(h0) | (bf16_bits(h1) << 16);
                lo[e / 2] = bf16_bits(l0) | (bf16_bits(l1) << 16);
            }
        }
        const int kb = k0 / MT_KBLK, c = (k0 % MT_KBLK) / 8;
        uint8_t* blk = xop + (size_t)kb * MT_XBLK;
        *(uint4*)(blk + n * 128 + ((c ^ (n & 7)) << 4)) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
        const int m = 16 + n;
        *(uint4*)(blk + m * 128 + ((c ^ (m & 7)) << 4)) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
    }
    ptx::fence_proxy_async_smem();
    __syncthreads();

    if (warp == 0) {
        if (lane == 0) {
            int issued = npre;
            for (int it = npre; it < total; ++it) {
                const int s = it % MT_STAGES, n = it / MT_STAGES;
                if (!ptx::mbar_wait_bounded(&empty[s], (n - 1) & 1, MT_WAIT_NS)) {
                    *flag = DEV_TIMEOUT_WEIGHTS;
                    break;
                }
                load(it);
                issued = it + 1;
            }
            // No copy into this CTA's shared memory is left in flight at exit: the last load of
            // every stage has landed (at once in the normal case, where the MMAs consumed it).
            for (int it = issued - MT_STAGES < 0 ? 0 : issued - MT_STAGES; it < issued; ++it)
                if (!ptx::mbar_wait_bounded(&full[it % MT_STAGES], (it / MT_STAGES) & 1, MT_WAIT_NS))
                    *flag = DEV_TIMEOUT_WEIGHTS;
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t IDESC = ptx::idesc_bf16_f32(MT_ROWS, MT_N);
            const uint32_t rbase = ptx::smem_u32(ring), xbase = ptx::smem_u32(xop);
            bool good = true;
            int it = 0;
            for (int j = 0; j < my_tiles; ++j) {
                const int buf = j & 1;
                if (j >= 2 && !ptx::mbar_wait_bounded(&acce[buf], ((j - 2) >> 1) & 1, MT_WAIT_NS)) good = false;
                ptx::tc_fence_after();
                const uint32_t acc = tmem + (uint32_t)(buf * MT_N);
                for (int kb = 0; kb < nkb; ++kb, ++it) {
                    const int s = it % MT_STAGES, n = it / MT_STAGES;
                    if (good && !ptx::mbar_wait_bounded(&full[s], n & 1, MT_WAIT_NS)) good = false;
                    ptx::tc_fence_after();
                    if (good) {
                        const uint32_t w = rbase + (uint32_t)(s * MT_WBYTES), x = xbase + (uint32_t)(kb * MT_XBLK);
#pragma unroll
                        for (int kk = 0; kk < MT_KBLK / 16; ++kk)
                            ptx::mma_bf16(acc, ptx::desc_sw128(w + kk * 32), ptx::desc_sw128(x + kk * 32), IDESC,
                                          (kb | kk) != 0);
                    }
                    ptx::mma_commit(&empty[s]);
                }
                // Committed even after a timeout so that the epilogue wakes up.
                ptx::mma_commit(&accf[buf]);
            }
            if (!good) *flag = DEV_TIMEOUT_MMA;
        }
    } else if (warp >= 4) {
        // TMEM lanes 32 (warp mod 4) .. + 31: weight row `row` of the tile.
        const int row = (warp & 3) * 32 + lane;
        const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
        for (int j = 0; j < my_tiles; ++j) {
            const int buf = j & 1;
            const int tile = t0 + j * dt;
            const bool ok = ptx::mbar_wait_bounded(&accf[buf], (j >> 1) & 1, MT_WAIT_NS);
            ptx::tc_fence_after();
            uint32_t h[16], l[16];
            ptx::tmem_ld_x16(lane_base + (uint32_t)(buf * MT_N), h);
            ptx::tmem_ld_x16(lane_base + (uint32_t)(buf * MT_N + 16), l);
            ptx::tmem_ld_wait();
            ptx::tc_fence_before();
            ptx::mbar_arrive(&acce[buf]);
            if (!ok) {
                if (lane == 0) *flag = DEV_TIMEOUT_MMA;
                continue;
            }
            const int r = tile * MT_ROWS + row;
            const float b = bias[r];
#pragma unroll
            for (int n = 0; n < 16; ++n)
                if (n < N) Y[(size_t)n * R + r] = (__uint_as_float(h[n]) + __uint_as_float(l[n])) + b;
        }
    }

    if (tid == 0 && *flag != 0) atomicCAS(err, 0, *flag);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc(tmem, 2 * MT_N);
}

}  // namespace

bool mod_tc_supported(const jpi_handle* h) {
    return h->tc && h->W % MT_KBLK == 0 && (mod_rows(h->L) * h->W) % MT_ROWS == 0 &&
           mod_tc_smem(h->W) + 1024 <= 227 * 1024;
}

jpi_status mod_tc_prepare(jpi_handle* h) {
    if (!mod_tc_supported(h)) return JPI_OK;
    const uint64_t R = (uint64_t)mod_rows(h->L) * h->W;
    JPI_TRY(tc_make_tmap(h->mod_w, R, h->W, MT_ROWS, &h->mod_map));
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_mod_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)(1024 + mod_tc_smem(h->W))));
    h->mod_tc = true;
    return JPI_OK;
}

jpi_status launch_mod_tc(jpi_handle* h, const float* X, float* Y, int N, cudaStream_t st) {
    const int R = mod_rows(h->L) * h->W;
    if (N < 1 || N > 16) {
        set_error("modulation pass of %d step times (1..16)", N);
        return JPI_ERR_INVALID_ARG;
    }
    const int ntiles = R / MT_ROWS;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(ntiles < h->num_sms ? ntiles : h->num_sms));
    cfg.blockDim = dim3(MT_THREADS);
    cfg.dynamicSmemBytes = 1024 + mod_tc_smem(h->W);
    cfg.stream = st;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr.val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = h->pdl ? 1 : 0;
    cudaError_t e = cudaLaunchKernelEx(&cfg, k_mod_tc, h->mod_map, X, (const float*)h->mod_b, Y, N, R,
                                       h->W, h->dev_err);
    if (e != cudaSuccess) {
        set_error("modulation launch failed: %s", cudaGetErrorString(e));
        return JPI_ERR_CUDA;
    }
    return JPI_OK;
}

}  // namespace jpi
