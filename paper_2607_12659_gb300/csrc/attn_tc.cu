// Attention of the suffix queries over [prefix KV ; suffix KV] with one shared KV head, on
// tensor cores (bf16 operands, fp32 accumulation and softmax).
//
// App. A of the paper: at every expert layer the queries come from the action-noise tokens
// (here the state token and the C action tokens) and the keys/values are the matching LLM
// layer's KV cache concatenated with the suffix tokens' own keys/values. With a single KV head
// every query head of every suffix token attends to the same K/V rows, so one request's
// S x H query rows form one dense [S*H][D] x [D][P+S] problem; rows are ordered token-major
// (row = i * H + head). The state row (i = 0) and the correction items' context rows
// (i < nctx) see the prefix and each other only.
//
// Grid: (32-row query blocks, key splits, requests). The key splits of one query block form a
// thread-block cluster. Inside a CTA, warp w takes query rows 16 (w mod 2) .. + 15 of every key
// block (staged in shared memory by bulk tensor copies): it computes the scores of key half w / 2, the
// two warps of a row group exchange their block maxima and write the probabilities P (bf16) to
// shared memory, and each then accumulates output columns half w / 2 over all keys of the block
// (one online softmax per row group, nothing left to merge). The cluster then
// combines the per-split (max, sum, output) triples through distributed shared memory in split
// order, so the result does not depend on timing. Each split pushes the rows owned by every other
// split into that split's dedicated receive buffer as soon as its own rows are final; the only
// cluster-wide waits are one before the first push (receive barriers initialised) and one before
// exit (every copy out of this CTA has landed).

#include "jpi_internal.h"
#include "ptx.h"
#include "tc_path.h"

#include <cooperative_groups.h>
#include <cstdlib>

namespace cg = cooperative_groups;

namespace jpi {
namespace {

constexpr int AT_ROWS = 32;      // query rows per CTA (2 row groups of 16)
constexpr int AT_KEYS = 64;      // keys per shared-memory block (2 halves of 32)
constexpr int AT_THREADS = 128;  // 4 warps: (row group, key half)
constexpr int AT_MAX_SPLITS = 16;
// Most rows one split receives: (splits - 1) x ceil(32 / splits), largest at 15 splits.
constexpr int AT_MAX_RECV_ROWS = 42;

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void mma16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
// 2^x by the hardware approximation (PTX ex2.approx.ftz.f32, relative error ~2^-22); the
// arguments here are <= 0 (differences to a running maximum).
__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

// Byte offset of 16-byte chunk `c` of row `r` of the query tile as its bulk tensor copies land
// it: D/64 column blocks of [32 rows][128 B], 16-byte chunks XOR-swizzled by (r mod 8).
__device__ __forceinline__ uint32_t q_off(int r, int c) {
    return (uint32_t)((c >> 3) * (AT_ROWS * 128) + r * 128 + (((c & 7) ^ (r & 7)) << 4));
}
// The same for a K or V block of KB rows (D/64 column blocks of [KB rows][128 B]).
template <int KB>
__device__ __forceinline__ uint32_t kv_off(int r, int c) {
    return (uint32_t)((c >> 3) * (KB * 128) + r * 128 + (((c & 7) ^ (r & 7)) << 4));
}

struct AttnArgs {
    int kv_row0;                // this layer's first row in the K/V tensor maps (all layers)
    __nv_bfloat16* o;           // [Mt][H * D]
    int S, H, P, kv_rows, chunk, nsplit;
    int nctx;                   // suffix rows 0..nctx-1 (state, context tokens) see P + nctx keys
    float scale_log2;           // log2(e) / sqrt(D)
    int* err;
};

// One exchanged partial row: D fp16 values of O, then m and l (fp32), padded to 16 bytes.
template <int D>
__host__ __device__ constexpr int attn_row_bytes() {
    return 2 * D + 16;
}
// Row stride (bytes) of the bf16 probability tile P [32][KB]: 16 bytes of padding put the 8 rows
// of an ldmatrix phase, and the 8 rows a warp's 4-byte stores hit, on disjoint banks.
template <int KB>
__host__ __device__ constexpr int AT_PSTRIDE() {
    return KB * 2 + 16;
}
// Shared-memory layout (bytes from the 128-aligned base): q and NBUF k/v buffers, reused after
// the key loop for this split's partial rows; the receive buffer; the P tile, block maxima and
// l shares; the receive barrier.
template <int D, int NBUF>
struct AttnSmem {
    static constexpr int KB = NBUF == 2 ? AT_KEYS / 2 : AT_KEYS;   // keys per block
    static constexpr int QKV = (AT_ROWS + 2 * KB * NBUF) * D * 2;
    static constexpr int OPART = 0;                              // [32][row bytes], after the keys
    static constexpr int REGION_USED = OPART + AT_ROWS * attn_row_bytes<D>();
    static constexpr int REGION = QKV > REGION_USED ? QKV : REGION_USED;
    static constexpr int RECV = REGION;                          // [AT_MAX_RECV_ROWS][row bytes]
    static constexpr int PB = RECV + AT_MAX_RECV_ROWS * attn_row_bytes<D>();   // [32][KB] bf16 P, padded rows
    static constexpr int XM = PB + AT_ROWS * AT_PSTRIDE<KB>();     // [2 halves][32] block maxima
    static constexpr int LS = XM + 2 * AT_ROWS * 4;                // [2 halves][32] l shares
    static constexpr int BAR = LS + 2 * AT_ROWS * 4;
    static constexpr int TOTAL = BAR + 32;   // receive, query, and NBUF K/V barriers
};

// NBUF = 2 when a split spans several key blocks: blocks of 32 keys, double-buffered (the next
// block's K/V loads are issued before the current block is processed) in the same shared memory
// as one 64-key block, so two CTAs still fit on an SM.
template <int D, int NBUF>
__global__ void __launch_bounds__(AT_THREADS) k_attn_tc(const __grid_constant__ CUtensorMap qmap,
                                                        const __grid_constant__ CUtensorMap kmap,
                                                        const __grid_constant__ CUtensorMap vmap,
                                                        const __grid_constant__ AttnArgs a) {
    using L = AttnSmem<D, NBUF>;
    constexpr int KB = L::KB;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (ptx::smem_u32(smem_raw) & 1023u)) & 1023u);
    uint8_t* qs = smem;                                  // [32][D] bf16
    uint8_t* ks = qs + AT_ROWS * D * 2;                  // [NBUF][k [64][D], v [64][D]] bf16
    uint8_t* vs = ks + KB * D * 2;
    constexpr uint32_t KV_BUF = 2 * KB * D * 2;     // bytes of one k/v buffer pair
    constexpr int ROWB = attn_row_bytes<D>();
    uint8_t* opart = smem + L::OPART;                    // [32][ROWB] this split's partial rows
    uint8_t* pbuf = smem + L::PB;                        // [32][KB] bf16 probabilities
    float* xmax = (float*)(smem + L::XM);                // [2][32] block maxima of each key half
    float* lsum = (float*)(smem + L::LS);                // [2][32] l of each key half
    uint8_t* recv = smem + L::RECV;                      // [(splits - 1) x rows_per][ROWB]
    uint64_t* rbar = (uint64_t*)(smem + L::BAR);
    uint64_t* qbar = rbar + 1;                           // the query tile's bulk copies
    uint64_t* kvbar = rbar + 2;                          // [NBUF] each K/V buffer's bulk copies

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int rg = warp & 1, kh = warp >> 1;             // row group, key half / column half
    const int rb = blockIdx.x, b = blockIdx.z;
    const int nrows = a.S * a.H, nk = a.P + a.S;
    const int row0 = rb * AT_ROWS;
    const int ns = a.nsplit;
    const int rank = (int)ptx::cluster_rank();           // == blockIdx.y (cluster spans the splits)
    const int k_begin = rank * a.chunk, k_end = min(nk, k_begin + a.chunk);
    // Rows [s * rows_per, ...) of the 32 belong to split s, which combines them.
    const int rows_per = (AT_ROWS + ns - 1) / ns;
    const int r_lo = min(AT_ROWS, rank * rows_per), r_hi = min(AT_ROWS, r_lo + rows_per);
    if (tid == 0) {
        ptx::mbar_init(rbar, 1);
        ptx::mbar_init(qbar, 1);
        for (int i = 0; i < NBUF; ++i) ptx::mbar_init(&kvbar[i], 1);
        ptx::fence_mbar_init();
        ptx::mbar_expect_tx(rbar, (uint32_t)((ns - 1) * (r_hi - r_lo) * ROWB));
    }
    __syncthreads();
    // Receive barriers are initialised cluster-wide before anyone pushes: arrive now, wait
    // before the first push (published by fence.mbarrier_init, so the arrival is relaxed).
    ptx::cluster_arrive_relaxed();

    // K and V blocks by bulk tensor copies (one thread): D/64 column blocks x KB/32 boxes of 32
    // rows each. Rows past the split's last key are whatever the store holds there (finite:
    // zero-initialised, or other requests' and layers' keys); their scores are masked.
    const uint32_t qs_u = ptx::smem_u32(qs), ks_u = ptx::smem_u32(ks), vs_u = ptx::smem_u32(vs);
    const int kv_row_b = a.kv_row0 + b * a.kv_rows;      // this request's key 0 in the maps
    const uint64_t pol = ptx::l2_policy_evict_first();
    auto load_block = [&](int key0, int buf) {
        uint8_t* kd = ks + buf * KV_BUF;
        uint8_t* vd = vs + buf * KV_BUF;
        ptx::mbar_expect_tx(&kvbar[buf], KV_BUF);
        for (int db = 0; db < D / 64; ++db)
            for (int hb = 0; hb < KB / 32; ++hb) {
                const uint32_t off = (uint32_t)(db * (KB * 128) + hb * (32 * 128));
                const int y = kv_row_b + key0 + hb * 32;
                ptx::tma_load_2d(kd + off, &kmap, &kvbar[buf], db * 64, y, pol);
                ptx::tma_load_2d(vd + off, &vmap, &kvbar[buf], db * 64, y, pol);
            }
    };
    // A first block made only of prefix keys (written before this graph ran) is fetched before
    // the dependency wait; one holding suffix keys (written by the QKV kernel) after it.
    const bool early = min(k_end, k_begin + KB) <= a.P;
    if (tid == 0) {
        ptx::prefetch_tmap(&qmap);
        if (early) load_block(k_begin, 0);
    }

    ptx::grid_dep_wait();

    // Query block: D/64 bulk tensor copies of 32 rows (rows past this request's S*H rows are
    // the next request's or zero fill; their results are never stored).
    if (tid == 0) {
        ptx::mbar_expect_tx(qbar, (uint32_t)(AT_ROWS * D * 2));
        for (int db = 0; db < D / 64; ++db)
            ptx::tma_load_2d(qs + db * (AT_ROWS * 128), &qmap, qbar, db * 64, b * nrows + row0, pol);
        if (!early) load_block(k_begin, 0);
    }

    // Per-thread rows g and g + 8 of this warp's 16; their visible key count.
    const int g = lane >> 2, cq = lane & 3;
    int nvis[2];
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
        const int R = row0 + rg * 16 + g + hh * 8;
        const int i = R / a.H;
        nvis[hh] = (R < nrows && i < a.nctx) ? a.P + a.nctx : nk;
    }

    // This warp's output columns: half kh of the D dimensions, for all keys of a block.
    constexpr int NOT = D / 16;                          // n-tiles of 8 columns per half
    float oacc[NOT][4];
#pragma unroll
    for (int n = 0; n < NOT; ++n) oacc[n][0] = oacc[n][1] = oacc[n][2] = oacc[n][3] = 0.f;
    // Both warps of a row group share one running maximum; l is this warp's key-half share.
    float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
    constexpr int HK = KB / 2;                      // keys per half
    const int ra = rg * 16 + g, rb2 = ra + 8;             // this thread's two rows
    const uint32_t pb_u = ptx::smem_u32(pbuf);

    int jb = 0;   // block index within the split
    for (int key0 = k_begin; key0 < k_end; key0 += KB, ++jb) {
        __syncthreads();   // every warp is done with the buffer refilled below (and with P)
        // Block jb sits in buffer jb mod NBUF (its (jb / NBUF)-th use); with two buffers the next
        // block is fetched into the other one while this one is processed.
        const int bi = NBUF == 2 ? (jb & 1) : 0;
        if (tid == 0) {
            if (NBUF == 2 && key0 + KB < k_end) load_block(key0 + KB, bi ^ 1);
            if (NBUF == 1 && key0 != k_begin) load_block(key0, 0);
        }
        const uint32_t par = NBUF == 2 ? ((jb >> 1) & 1) : (jb & 1);
        bool landed = ptx::mbar_wait_bounded(&kvbar[bi], par, 200ull * 1000 * 1000);
        if (key0 == k_begin) landed = ptx::mbar_wait_bounded(qbar, 0, 200ull * 1000 * 1000) && landed;
        if (!landed && tid == 0) atomicCAS(a.err, 0, (int)DEV_TIMEOUT_WEIGHTS);
        const uint32_t kbuf_u = ks_u + bi * KV_BUF, vbuf_u = vs_u + bi * KV_BUF;

        // S = Q K^T for this warp's 16 rows x its key half.
        float sacc[HK / 8][4];
#pragma unroll
        for (int n = 0; n < HK / 8; ++n) sacc[n][0] = sacc[n][1] = sacc[n][2] = sacc[n][3] = 0.f;
#pragma unroll
        for (int kc = 0; kc < D / 16; ++kc) {
            uint32_t a0, a1, a2, a3;
            {
                const int r = rg * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
                const int c = kc * 2 + (lane >> 4);
                ldsm_x4(qs_u + q_off(r, c), a0, a1, a2, a3);
            }
#pragma unroll
            for (int nt = 0; nt < HK / 8; nt += 2) {
                uint32_t b0, b1, b2, b3;
                const int r = kh * HK + (nt + (lane >> 4)) * 8 + (lane & 7);
                const int c = kc * 2 + ((lane >> 3) & 1);
                ldsm_x4(kbuf_u + kv_off<KB>(r, c), b0, b1, b2, b3);
                mma16816(sacc[nt], a0, a1, a2, a3, b0, b1);
                mma16816(sacc[nt + 1], a0, a1, a2, a3, b2, b3);
            }
        }
        // Scale to log2 units, mask; the block maximum of each row over both key halves.
        float bmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
        for (int nt = 0; nt < HK / 8; ++nt)
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int key = key0 + kh * HK + nt * 8 + 2 * cq + (e & 1);
                const int hh = e >> 1;
                const float s = (key < k_end && key < nvis[hh]) ? sacc[nt][e] * a.scale_log2 : -INFINITY;
                sacc[nt][e] = s;
                bmax[hh] = fmaxf(bmax[hh], s);
            }
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            bmax[hh] = fmaxf(bmax[hh], __shfl_xor_sync(0xffffffffu, bmax[hh], 1));
            bmax[hh] = fmaxf(bmax[hh], __shfl_xor_sync(0xffffffffu, bmax[hh], 2));
        }
        if (cq == 0) {
            xmax[kh * AT_ROWS + ra] = bmax[0];
            xmax[kh * AT_ROWS + rb2] = bmax[1];
        }
        ptx::named_bar_sync(1 + rg, 64);   // the two warps of this row group
        bmax[0] = fmaxf(bmax[0], xmax[(1 - kh) * AT_ROWS + ra]);
        bmax[1] = fmaxf(bmax[1], xmax[(1 - kh) * AT_ROWS + rb2]);
        float alpha[2], mnew[2];
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            mnew[hh] = fmaxf(m_run[hh], bmax[hh]);
            alpha[hh] = (mnew[hh] == -INFINITY) ? 1.f : fast_exp2(m_run[hh] - mnew[hh]);
        }
        // P = 2^(s - m) for this warp's keys: summed into l, stored as bf16 for both warps' P V.
        float psum[2] = {0.f, 0.f};
#pragma unroll
        for (int nt = 0; nt < HK / 8; ++nt) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int hh = e >> 1;
                const float p = (sacc[nt][e] == -INFINITY) ? 0.f : fast_exp2(sacc[nt][e] - mnew[hh]);
                sacc[nt][e] = p;
                psum[hh] += p;
            }
            const uint32_t col_b = (uint32_t)(kh * HK + nt * 8 + 2 * cq) * 2;
            *(uint32_t*)(pbuf + ra * AT_PSTRIDE<KB>() + col_b) = pack_bf16x2(sacc[nt][0], sacc[nt][1]);
            *(uint32_t*)(pbuf + rb2 * AT_PSTRIDE<KB>() + col_b) = pack_bf16x2(sacc[nt][2], sacc[nt][3]);
        }
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            psum[hh] += __shfl_xor_sync(0xffffffffu, psum[hh], 1);
            psum[hh] += __shfl_xor_sync(0xffffffffu, psum[hh], 2);
            l_run[hh] = l_run[hh] * alpha[hh] + psum[hh];
            m_run[hh] = mnew[hh];
        }
#pragma unroll
        for (int n = 0; n < NOT; ++n) {
            oacc[n][0] *= alpha[0];
            oacc[n][1] *= alpha[0];
            oacc[n][2] *= alpha[1];
            oacc[n][3] *= alpha[1];
        }
        ptx::named_bar_sync(1 + rg, 64);   // both halves of P are in shared memory
        // O[:, half kh] += P V over all KB keys of the block.
#pragma unroll
        for (int j = 0; j < KB / 16; ++j) {
            uint32_t a0, a1, a2, a3;
            {
                const int r = rg * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
                const int c = j * 2 + (lane >> 4);
                ldsm_x4(pb_u + (uint32_t)(r * AT_PSTRIDE<KB>() + c * 16), a0, a1, a2, a3);
            }
#pragma unroll
            for (int dt = 0; dt < NOT; dt += 2) {
                uint32_t b0, b1, b2, b3;
                const int r = j * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
                const int c = kh * NOT + dt + (lane >> 4);
                ldsm_x4_t(vbuf_u + kv_off<KB>(r, c), b0, b1, b2, b3);
                mma16816(oacc[dt], a0, a1, a2, a3, b0, b1);
                mma16816(oacc[dt + 1], a0, a1, a2, a3, b2, b3);
            }
        }
    }

    // ---- this split's partial rows (q/k/v are dead past this barrier) ----
    if (cq == 0) {
        lsum[kh * AT_ROWS + ra] = l_run[0];
        lsum[kh * AT_ROWS + rb2] = l_run[1];
    }
    __syncthreads();
    {
        // O unnormalised in fp16 (a value beyond the fp16 range raises a device error), then
        // m and l in fp32; each warp writes its half of the columns.
        if (kh == 0 && cq == 0) {
            *(float2*)(opart + ra * ROWB + 2 * D) = make_float2(m_run[0], lsum[ra] + lsum[AT_ROWS + ra]);
            *(float2*)(opart + rb2 * ROWB + 2 * D) = make_float2(m_run[1], lsum[rb2] + lsum[AT_ROWS + rb2]);
        }
        bool range_ok = true;
#pragma unroll
        for (int n = 0; n < NOT; ++n) {
            const int col = kh * (D / 2) + n * 8 + 2 * cq;
            range_ok &= fabsf(oacc[n][0]) <= 65000.f && fabsf(oacc[n][1]) <= 65000.f &&
                        fabsf(oacc[n][2]) <= 65000.f && fabsf(oacc[n][3]) <= 65000.f;
            *(__half2*)(opart + ra * ROWB + col * 2) = __floats2half2_rn(oacc[n][0], oacc[n][1]);
            *(__half2*)(opart + rb2 * ROWB + col * 2) = __floats2half2_rn(oacc[n][2], oacc[n][3]);
        }
        if (!range_ok) atomicCAS(a.err, 0, (int)DEV_FP16_RANGE);
    }
    ptx::fence_proxy_async_smem();
    __syncthreads();

    // ---- exchange: push every other split's rows into its receive buffer ----
    ptx::cluster_wait();
    // Lane s of warp 0 sends split s its rows (the copies to all splits issue together).
    if (warp == 0 && lane < ns && lane != rank) {
        const int s = lane;
        const int lo = min(AT_ROWS, s * rows_per), hi = min(AT_ROWS, lo + rows_per);
        if (hi > lo) {
            const uint32_t bar_u = ptx::smem_u32(rbar);
            const int slot = rank < s ? rank : rank - 1;   // split s stores senders != s in order
            const uint32_t dst = ptx::smem_u32(recv + (size_t)slot * rows_per * ROWB);
            ptx::bulk_copy_to_cluster(ptx::dsmem_map(dst, (uint32_t)s), opart + (size_t)lo * ROWB,
                                      (uint32_t)((hi - lo) * ROWB), ptx::dsmem_map(bar_u, (uint32_t)s));
        }
    }
    const bool got = ptx::mbar_wait_bounded(rbar, 0, 200ull * 1000 * 1000);
    // Everything addressed to this split has landed (seen through its own barrier); once all
    // splits arrive, every copy out of this CTA has landed too.
    ptx::cluster_arrive_relaxed();
    // The next kernel may start now (its weight prefetch no longer competes with this one's
    // loads and exchange).
    ptx::grid_dep_launch();
    // Row r of split s: this CTA's own partial, or the slice split s sent.
    auto srow = [&](int s, int r) -> const uint8_t* {
        if (s == rank) return opart + (size_t)r * ROWB;
        const int slot = s < rank ? s : s - 1;
        return recv + ((size_t)slot * rows_per + (r - r_lo)) * ROWB;
    };

    // ---- combine the splits for the owned rows, in split order ----
    // One warp per owned row: lane s (and s + 16) turns split s's (m, l) into its coefficient
    // w_s / L by butterflies over the 16 splits; each lane then sums 8 output dimensions over the
    // splits in split order, taking the coefficients by shuffles.
    const int nrow_here = r_hi - r_lo;
    for (int rr = warp; rr < nrow_here; rr += AT_THREADS / 32) {
        const int r = r_lo + rr;
        const int sl = lane & (AT_MAX_SPLITS - 1);
        const float2 ml = sl < ns ? *(const float2*)(srow(sl, r) + 2 * D) : make_float2(-INFINITY, 0.f);
        float mx = ml.x;
#pragma unroll
        for (int o = 1; o < AT_MAX_SPLITS; o <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        const float w = (ml.x == -INFINITY) ? 0.f : fast_exp2(ml.x - mx);
        float L = w * ml.y;
#pragma unroll
        for (int o = 1; o < AT_MAX_SPLITS; o <<= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
        const float cf = L > 0.f ? w / L : 0.f;   // 0 for lanes past the last split
        const int R = row0 + r, d = lane * 8;
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        // All 16 slots are loaded together (slots past the last split read this CTA's own row
        // with a zero coefficient), then summed in split order.
#pragma unroll
        for (int s = 0; s < AT_MAX_SPLITS; ++s) {
            const float c = __shfl_sync(0xffffffffu, cf, s);
            if (d < D) {
                const uint4 hv = *(const uint4*)(srow(s < ns ? s : rank, r) + 2 * d);
                const uint32_t w4[4] = {hv.x, hv.y, hv.z, hv.w};
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const float2 v = __half22float2(*reinterpret_cast<const __half2*>(&w4[k]));
                    acc[2 * k] = fmaf(c, v.x, acc[2 * k]);
                    acc[2 * k + 1] = fmaf(c, v.y, acc[2 * k + 1]);
                }
            }
        }
        if (d < D && R < nrows && got) {
            const int i = R / a.H, head = R - i * a.H;
            const size_t tok = (size_t)b * a.S + i;
            *(uint4*)(a.o + (tok * a.H + head) * D + d) =
                make_uint4(pack_bf16x2(acc[0], acc[1]), pack_bf16x2(acc[2], acc[3]), pack_bf16x2(acc[4], acc[5]),
                           pack_bf16x2(acc[6], acc[7]));
        }
    }
    if (tid == 0 && !got) atomicCAS(a.err, 0, (int)DEV_TIMEOUT_MMA);
    // No split exits while a copy out of its shared memory may still be in flight.
    ptx::cluster_wait();
}

template <int D, int NBUF>
size_t attn_smem() {
    return 1024 + (size_t)AttnSmem<D, NBUF>::TOTAL;
}

template <int D>
jpi_status launch_attn_d(jpi_handle* h, int l, int B, int C, cudaStream_t st) {
    const int S = C + h->n_ctx(), nrows = S * h->H, nk = h->cur_prefix + S;
    const int rblocks = (nrows + AT_ROWS - 1) / AT_ROWS;
    // Key splits: the largest power of two that keeps the launch within two CTAs per SM, at
    // most 16 (one cluster): 16 asked (14 after rounding the chunk to whole 64-key blocks) for one
    // pi0.5-shaped request, 8 for two, 4 for three to five, one when many requests fill the GPU by
    // themselves (then each CTA runs an online softmax over all keys and nothing is exchanged).
    // Clusters of a power of two measured faster than the counts in between (batch 4: 4 splits
    // 13.9 us, 3 splits 18.2, 6 splits 19.7 per launch; batch 2: 8 splits 9.3, 12 splits 13.0).
    // The split follows the launch's sizes, so a request's low-order bits depend on the batch
    // size it runs with; they never depend on timing.
    // In the batch-invariant mode the split is the one a single request gets, whatever B.
    const int blocks = rblocks * (h->batch_invariant ? 1 : B);
    int want = 1;
    while (2 * want <= AT_MAX_SPLITS && (long long)blocks * want * 2 <= 2LL * h->num_sms) want *= 2;
    // A split count asked through the environment at create time replaces that choice.
    if (h->attn_force_splits > 0) want = h->attn_force_splits;
    want = want < 1 ? 1 : (want > h->attn_max_splits ? h->attn_max_splits : want);
    int chunk = (nk + want - 1) / want;
    chunk = (chunk + 15) / 16 * 16;
    const int ns = (nk + chunk - 1) / chunk;
    AttnArgs a;
    a.kv_row0 = l * h->maxB * h->kv_rows;
    a.o = (__nv_bfloat16*)h->o;
    a.S = S;
    a.nctx = h->n_ctx();
    a.H = h->H;
    a.P = h->cur_prefix;
    a.kv_rows = h->kv_rows;
    a.chunk = chunk;
    a.nsplit = ns;
    a.scale_log2 = 1.4426950408889634f / sqrtf((float)D);
    a.err = h->dev_err;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(rblocks, ns, B);
    cfg.blockDim = dim3(AT_THREADS);
    // Splits of 2..8 key blocks: 32-key blocks, double-buffered (measured faster there); longer
    // splits keep 64-key blocks, where the per-block rescale of the output accumulators would
    // otherwise double.
    const bool two = chunk > AT_KEYS && chunk <= 8 * AT_KEYS;
    cfg.dynamicSmemBytes = two ? attn_smem<D, 2>() : attn_smem<D, 1>();
    cfg.stream = st;
    cudaLaunchAttribute attrs[2];
    int n = 0;
    attrs[n].id = cudaLaunchAttributeClusterDimension;
    attrs[n].val.clusterDim.x = 1;
    attrs[n].val.clusterDim.y = ns;
    attrs[n].val.clusterDim.z = 1;
    ++n;
    if (h->pdl) {
        attrs[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attrs[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    cfg.attrs = attrs;
    cfg.numAttrs = n;
    cudaError_t e = two ? cudaLaunchKernelEx(&cfg, k_attn_tc<D, 2>, h->qmap_at, h->kmap_at, h->vmap_at, a)
                        : cudaLaunchKernelEx(&cfg, k_attn_tc<D, 1>, h->qmap_at, h->kmap_at, h->vmap_at, a);
    if (e != cudaSuccess) {
        set_error("attention launch failed: %s", cudaGetErrorString(e));
        return JPI_ERR_CUDA;
    }
    return JPI_OK;
}

template <int D>
jpi_status prepare_d(jpi_handle* h) {
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_attn_tc<D, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)attn_smem<D, 1>()));
    JPI_CUDA_TRY(cudaFuncSetAttribute(k_attn_tc<D, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)attn_smem<D, 2>()));
    if (cudaFuncSetAttribute(k_attn_tc<D, 1>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess ||
        cudaFuncSetAttribute(k_attn_tc<D, 2>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
        cudaGetLastError();
        h->attn_max_splits = 8;
    } else {
        h->attn_max_splits = AT_MAX_SPLITS;
    }
    return JPI_OK;
}

}  // namespace

bool attn_tc_supported(const jpi_handle* h) {
    return h->D == 64 || h->D == 128 || h->D == 256;
}

jpi_status attn_tc_prepare(jpi_handle* h) {
    // JPI_ATTN_SPLITS fixes the number of key splits (clamped to 1 .. the largest cluster),
    // so that results can be compared across split counts; unset, the launch chooses.
    const char* env = std::getenv("JPI_ATTN_SPLITS");
    h->attn_force_splits = env ? std::atoi(env) : 0;
    // The query tile as 32-row boxes of 64 columns (128-byte swizzle) over q [maxMt * H][D].
    JPI_TRY(tc_make_tmap(h->q, (uint64_t)h->maxMt * h->H, h->D, AT_ROWS, &h->qmap_at));
    // K and V of all layers [L * maxB * kv_rows][D] as 32-row boxes.
    const uint64_t kv_rows_all = (uint64_t)h->L * h->maxB * h->kv_rows;
    JPI_TRY(tc_make_tmap(h->kv_k, kv_rows_all, h->D, 32, &h->kmap_at));
    JPI_TRY(tc_make_tmap(h->kv_v, kv_rows_all, h->D, 32, &h->vmap_at));
    switch (h->D) {
        case 64: return prepare_d<64>(h);
        case 128: return prepare_d<128>(h);
        case 256: return prepare_d<256>(h);
        default:
            set_error("attention head_dim %d is not tiled", h->D);
            return JPI_ERR_UNSUPPORTED;
    }
}

jpi_status launch_attn_tc(jpi_handle* h, int l, int B, int C, cudaStream_t st) {
    switch (h->D) {
        case 64: return launch_attn_d<64>(h, l, B, C, st);
        case 128: return launch_attn_d<128>(h, l, B, C, st);
        case 256: return launch_attn_d<256>(h, l, B, C, st);
        default:
            set_error("attention head_dim %d is not tiled", h->D);
            return JPI_ERR_UNSUPPORTED;
    }
}

}  // namespace jpi
