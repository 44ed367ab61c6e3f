// Large-M projection kernel for batched denoises (included by tc_path.cu, inside jpi's anonymous
// namespace), used when a launch has enough tokens to fill the GPU without splitting K.
//
// Output tile = one 128-row weight tile x one 128-row operand tile (128 tokens, or for the
// RMSNorm-fed kinds two 64-row tiles of 63 tokens + one beta row) over the whole K range. At
// large batch these projections are bound by the rate at which one SM takes operands in from
// L2 (87-100 GB/s measured per SM), not by the MMAs.
// Persistent: one CTA per SM walks the tiles u = blockIdx.x, + gridDim.x, ... (weight tile
// fastest), and its roles overlap consecutive tiles:
//   warp 0  one thread streams (weight block, operand block) pairs by bulk tensor copies into a
//           ring of STAGES shared-memory stages (full/empty mbarriers), tile after tile;
//   warp 1  one thread issues the tcgen05.mma chain (M = 128, N = 128, K = 16 each) of a tile
//           into one of two TMEM accumulators (tile j into buffer j mod 2, once the epilogue has
//           read tile j - 2 out of it) and releases each stage through tcgen05.commit;
//   warps 2-9  the epilogue, two groups of four warps (group g takes accumulator columns
//           64g..64g+63, one TMEM lane = weight row per thread). Every global input of a tile
//           (residual rows, rotary factors, the norm's sums of squares) is fetched before the
//           accumulator is waited for, all loads in flight together, so their latency hides
//           behind the MMAs (fetched in dependent chunks after it, it made the epilogue as long
//           as the tile's operand stream); one thread waits for the accumulator and the others
//           at a named barrier. Residual kinds copy the residual rows of the tile into a shared fp32
//           tile [token][feature] with 16-byte async copies, add their accumulator rows into it,
//           then write the new residual, the next norm's operand and each token's sum of squares
//           a token row per warp instruction (16 / 8 bytes per lane). The RMSNorm-fed kinds copy
//           their accumulator to a shared staging tile [row][token] where the row pairs
//           (p, p + 64) of rotary / GeGLU meet. After the read-out the TMEM buffer goes back to
//           the MMA thread.
// The next kernel is released once this CTA's last accumulator is complete. All waits are
// bounded.

constexpr int BIG_NT = 128;                       // operand rows per tile
constexpr int BIG_EPI = 256;                     // epilogue threads: two groups of 4 warps
constexpr int BIG_THREADS = 64 + BIG_EPI;
constexpr int BIG_XBYTES = BIG_NT * KBLK * 2;     // 16 KB operand block
constexpr int BIG_STAGE_BYTES = TILE_BYTES + BIG_XBYTES;
constexpr int BIG_YS = BIG_NT + 1;                // [row][token] staging stride: conflict-free rows and columns
constexpr int BIG_HS = BIG_NT + 4;                // [token][feature] residual stride: 16-byte rows
constexpr int BIG_YBYTES = BIG_NT * BIG_HS * 4;   // room for either layout

// S CTAs of a cluster split the K range of each unit (S = 1: no split). Each CTA then owns
// TOK = 128 / S of the unit's tokens: it sends the fp32 partial of every other CTA's tokens to that
// CTA ([token][feature] slices, one bulk copy per peer) and sums the S partials of its own tokens in
// rank order. The exchange buffers take shared memory from the ring, which keeps 3 (S = 2, 4) or
// 2 (S = 8) stages of 32 KB in flight.
template <int S>
struct BigCfg {
    static constexpr int STAGES = S == 1 ? 4 : (S == 8 ? 2 : 3);
    static constexpr int TOK = BIG_NT / S;                                 // tokens owned per CTA
    static constexpr int SLICE = TOK * BIG_NT * 4;                         // one [TOK][128] fp32 slice
    static constexpr int YBYTES = S == 1 ? BIG_YBYTES : TOK * BIG_HS * 4;  // staging tile
    static constexpr int SEND = (S - 1) * SLICE;                           // outgoing slices
    static constexpr int RECV = S == 1 ? 0 : S * SLICE;                    // partials by rank (own one too)
};

template <int S>
__host__ __device__ constexpr int big_smem_bytes() {
    // stages | staging tile | send | recv | rinv[128] | bars (full, empty, acc full[2], acc empty[2],
    // recv full, peers free) + TMEM slot + flag
    return BigCfg<S>::STAGES * BIG_STAGE_BYTES + BigCfg<S>::YBYTES + BigCfg<S>::SEND + BigCfg<S>::RECV +
           BIG_NT * 4 + 160;
}

template <int KIND, int S>
__global__ void __launch_bounds__(BIG_THREADS, 1) k_tc_gemm_big(const __grid_constant__ CUtensorMap wmap,
                                                             const __grid_constant__ CUtensorMap xmap,
                                                             const __grid_constant__ GemmArgs a) {
    using CF = BigCfg<S>;
    constexpr int STAGES = CF::STAGES;
    constexpr int TOK = CF::TOK;
    constexpr bool NORM_IN = (KIND == G_QKV || KIND == G_GU);
    static_assert(S == 1 || !NORM_IN, "the K split serves the residual kinds");
    constexpr int TT = NORM_IN ? 2 * XS_TOKENS : BIG_NT;   // tokens per tile
    constexpr uint32_t IDESC = ptx::idesc_bf16_f32(TILE_ROWS, BIG_NT);

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (ptx::smem_u32(smem_raw) & 1023u)) & 1023u);
    uint8_t* stages = smem;                                             // [stage][W 16 KB | X 16 KB]
    float* ystage = (float*)(smem + STAGES * BIG_STAGE_BYTES);          // staging tile
    float* sendb = (float*)((uint8_t*)ystage + CF::YBYTES);             // [S - 1][TOK][128] to the peers
    float* recvb = (float*)((uint8_t*)sendb + CF::SEND);                // [S][TOK][128] by sender rank
    float* rinv_s = (float*)((uint8_t*)recvb + CF::RECV);               // [128] column scales (norm-fed kinds)
    uint64_t* full = (uint64_t*)(rinv_s + BIG_NT);
    uint64_t* empty = full + STAGES;
    uint64_t* accf = empty + STAGES;   // [2] accumulator buffer holds a finished tile
    uint64_t* acce = accf + 2;         // [2] the epilogue has read it out
    uint64_t* recvf = acce + 2;        // the peers' slices of this unit have landed
    uint64_t* pfree = recvf + 1;       // every peer has summed the slices of the last unit
    uint32_t* tmem_slot = (uint32_t*)(pfree + 1);
    int* flag = (int*)(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int rank = S == 1 ? 0 : (int)ptx::cluster_rank();
    const int nkb = a.nkb / S;                 // K blocks of this CTA
    const int kb0 = rank * nkb;
    const int ntiles = a.ntiles;
    const int nxt = (a.Mt + TT - 1) / TT;
    const int total = ntiles * nxt;
    const int u0 = (int)blockIdx.x / S, du = (int)gridDim.x / S;

    if (warp == 1) {
        ptx::tmem_alloc(tmem_slot, 2 * BIG_NT);
        ptx::tmem_relinquish();
    }
    if (tid == 0) {
        for (int i = 0; i < STAGES; ++i) {
            ptx::mbar_init(&full[i], 1);
            ptx::mbar_init(&empty[i], 1);
        }
        ptx::mbar_init(&accf[0], 1);
        ptx::mbar_init(&accf[1], 1);
        ptx::mbar_init(&acce[0], BIG_EPI);
        ptx::mbar_init(&acce[1], BIG_EPI);
        ptx::mbar_init(recvf, 1);
        ptx::mbar_init(pfree, S > 1 ? S - 1 : 1);
        ptx::fence_mbar_init();
        *flag = 0;
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    // Split K: every CTA of the cluster has initialised its barriers before any peer aims a copy or
    // an arrival at them.
    if (S > 1) ptx::cluster_sync_all();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            const uint64_t pol = ptx::l2_policy_evict_first();
            auto load_w = [&](int tile, int kb, int s) {
                ptx::mbar_expect_tx(&full[s], (uint32_t)BIG_STAGE_BYTES);
                ptx::tma_load_2d(stages + s * BIG_STAGE_BYTES, &wmap, &full[s], 0, (tile * a.nkb + kb0 + kb) * TILE_ROWS,
                                 pol);
            };
            ptx::prefetch_tmap(&xmap);
            auto load_x = [&](int xt, int kb, int s) {
                uint8_t* xs = stages + s * BIG_STAGE_BYTES + TILE_BYTES;
                ptx::tma_load_2d(xs, &xmap, &full[s], (kb0 + kb) * KBLK, xt * BIG_NT, pol);
                ptx::tma_load_2d(xs + XBLK_BYTES, &xmap, &full[s], (kb0 + kb) * KBLK, xt * BIG_NT + NT, pol);
            };
            // Weight blocks of the first tile's first stages do not depend on the previous kernel.
            const int npre = u0 < total ? (nkb < STAGES ? nkb : STAGES) : 0;
            for (int kb = 0; kb < npre; ++kb) load_w(u0 % ntiles, kb, kb);
            ptx::grid_dep_wait();
            int it = 0;   // k-block counter over this CTA's tiles: stage it mod STAGES
            bool ok = true;
            for (int u = u0; u < total && ok; u += du) {
                const int tile = u % ntiles, xt = u / ntiles;
                for (int kb = 0; kb < nkb; ++kb, ++it) {
                    const int s = it % STAGES, n = it / STAGES;
                    if (it < npre) {   // first tile, weights already in flight
                        load_x(xt, kb, s);
                        continue;
                    }
                    if (it >= STAGES && !ptx::mbar_wait_bounded(&empty[s], (n - 1) & 1, WAIT_LIMIT_NS)) {
                        *flag = DEV_TIMEOUT_WEIGHTS;
                        ok = false;
                        break;
                    }
                    load_w(tile, kb, s);
                    load_x(xt, kb, s);
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t base = ptx::smem_u32(stages);
            bool good = true;
            int it = 0;
            for (int u = u0, j = 0; u < total; u += du, ++j) {
                const int buf = j & 1;
                // Tile j - 2 has been read out of this accumulator buffer.
                if (j >= 2 && !ptx::mbar_wait_bounded(&acce[buf], ((j - 2) >> 1) & 1, WAIT_LIMIT_NS)) good = false;
                ptx::tc_fence_after();
                const uint32_t acc = tmem + (uint32_t)(buf * BIG_NT);
                for (int kb = 0; kb < nkb; ++kb, ++it) {
                    const int s = it % STAGES, n = it / STAGES;
                    if (good && !ptx::mbar_wait_bounded(&full[s], n & 1, WAIT_LIMIT_NS)) good = false;
                    ptx::tc_fence_after();
                    if (good) {
                        const uint32_t w = base + s * BIG_STAGE_BYTES, x = w + TILE_BYTES;
#pragma unroll
                        for (int kk = 0; kk < KBLK / 16; ++kk)
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
    } else {
        // ---- epilogue: TMEM lane `row` (weight row) of the accumulator per thread ----
        const int et = (tid - 64) & 127, eg = (tid - 64) >> 7;   // thread within its group, group
        const int row = (warp & 3) * 32 + lane;
        ptx::grid_dep_wait();
        // Norm-fed kinds: thread (pair p, token half h) of the staging tile, tokens j_lo.. of the half.
        const int p = et & 63, h = et >> 6;
        const int j_lo = 32 * eg, nj = eg ? XS_TOKENS - 32 : 32;
        bool ok = true;
        // A tile's global inputs, all loads in flight together: the residual rows of the tile's
        // tokens (residual kinds: epilogue warp ew copies tokens 16 ew.. into the shared tile
        // [token][feature], 16 bytes per lane), or the rotary factors of this thread's tokens (QKV).
        const int ew = (tid - 64) >> 5;
        float2 cs[32];
        float gam = 0.f;
        float4 sg4 = make_float4(0.f, 0.f, 0.f, 0.f);   // next norm's scale of features 4 lane..
        auto fetch = [&](int tile, int tok0) {
            if constexpr (!NORM_IN) {
                const int f0 = tile * TILE_ROWS;
                gam = a.gamma[f0 + row];
                if (a.xs) sg4 = *(const float4*)(a.sigma_next + f0 + 4 * lane);
#pragma unroll
                for (int k = 0; k < TOK / 8; ++k) {
                    const int c = (TOK / 8) * ew + k, t = tok0 + rank * TOK + c;
                    const bool in = t < a.Mt;
                    ptx::cp_async_16(ptx::smem_u32(ystage + c * BIG_HS + 4 * lane),
                                     a.hres + (in ? (size_t)t * a.W + f0 + 4 * lane : 0), in);
                }
            } else if constexpr (KIND == G_QKV) {
                const int hd = a.D >> 1;
                const int pair = tile * 64 + p;
                const int sec = pair / hd, d = pair - sec * hd;
                const bool rot = a.rope && sec <= a.H;
                const int tfirst = tok0 + h * XS_TOKENS + j_lo;
                int ql = tfirst % a.S;   // position of the token in its request
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const bool in = rot && i < nj && tfirst + i < a.Mt;
                    cs[i] = in ? __ldg(a.rope + (size_t)(a.P + ql) * hd + d) : make_float2(1.f, 0.f);
                    if (++ql == a.S) ql = 0;
                }
            }
        };
        for (int u = u0, j = 0; u < total; u += du, ++j) {
            const int buf = j & 1;
            const int tile = u % ntiles, xt = u / ntiles;
            const int tok0 = xt * TT;
            if (NORM_IN && eg == 0) {
                // Column scale: rinv of the column's token from the sums of squares (added in slot
                // order, loaded 8 at a time), 1 for the beta columns 63 and 127.
                const int c = et;
                const int t = tok0 + (c >> 6) * XS_TOKENS + (c & 63);
                float r = 1.f;
                if ((c & 63) != 63) {
                    r = 0.f;
                    if (t < a.Mt) {
                        float s = 0.f;
                        for (int s0 = 0; s0 < a.nslot; s0 += 8) {
                            float v[8];
#pragma unroll
                            for (int k = 0; k < 8; ++k)
                                v[k] = s0 + k < a.nslot ? a.ss[(size_t)(s0 + k) * a.ss_ld + t] : 0.f;
#pragma unroll
                            for (int k = 0; k < 8; ++k) s += v[k];
                        }
                        r = rsqrtf(s * a.inv_w + a.eps);
                    }
                }
                rinv_s[c] = r;
            }
            fetch(tile, tok0);
            if (!NORM_IN) ptx::cp_async_wait_all();
            // Split K: every peer has summed the last unit's slices, so this CTA's outgoing slices
            // (read by those copies) and the peers' receive slots are free again.
            if (S > 1 && tid == 64 && j > 0 && !ptx::mbar_wait_cluster_bounded(pfree, (j - 1) & 1, WAIT_LIMIT_NS))
                *flag = DEV_TIMEOUT_MMA;
            if (tid == 64 && !ptx::mbar_wait_bounded(&accf[buf], (j >> 1) & 1, WAIT_LIMIT_NS)) *flag = DEV_TIMEOUT_MMA;
            // rinv or the residual rows published; the MMAs of the tile are done.
            ptx::named_bar_sync(1, BIG_EPI);
            ptx::tc_fence_after();
            // This CTA's last accumulator is complete: the next kernel may start streaming its weights.
            if (u + du >= total) ptx::grid_dep_launch();
            ok = ok && *flag == 0;
            {
                const uint32_t lane_base = tmem + (uint32_t)(buf * BIG_NT) + ((uint32_t)((warp & 3) * 32) << 16);
                if constexpr (NORM_IN) {
                    // Accumulator row -> staging row: y = rinv * acc + W beta of the column's
                    // 64-group (column 64 eg + 63 holds W beta).
                    float beta;
                    {
                        uint32_t r0[16];
                        ptx::tmem_ld_x16(lane_base + (uint32_t)(64 * eg + 48), r0);
                        ptx::tmem_ld_wait();
                        beta = __uint_as_float(r0[15]);
                    }
#pragma unroll
                    for (int c0 = 64 * eg; c0 < 64 * eg + 64; c0 += 32) {
                        uint32_t r[2][16];
                        ptx::tmem_ld_x16(lane_base + (uint32_t)c0, r[0]);
                        ptx::tmem_ld_x16(lane_base + (uint32_t)(c0 + 16), r[1]);
                        ptx::tmem_ld_wait();
#pragma unroll
                        for (int hh = 0; hh < 2; ++hh)
#pragma unroll
                            for (int i = 0; i < 16; ++i) {
                                const int c = c0 + 16 * hh + i;
                                const float v = __uint_as_float(r[hh][i]);
                                ystage[row * BIG_YS + c] = (c & 63) == 63 ? 0.f : rinv_s[c] * v + beta;
                            }
                    }
                    ptx::tc_fence_before();
                    ptx::mbar_arrive(&acce[buf]);
                    ptx::named_bar_sync(1, BIG_EPI);   // staging rows of the pair partners written
                    // Rows p and p + 64 of this tile for this thread's tokens of half h.
                    const int pair = tile * 64 + p;
                    int sec = 0, d = 0;
                    if (KIND == G_QKV) {
                        const int hd = a.D >> 1;
                        sec = pair / hd;
                        d = pair - sec * hd;
                    }
                    const bool rot = KIND == G_QKV && a.rope && sec <= a.H;
                    const int tfirst = tok0 + h * XS_TOKENS + j_lo;
                    int qb = tfirst / a.S, qi = tfirst - qb * a.S;   // request and position of the token
#pragma unroll
                    for (int jj = 0; jj < 32; ++jj) {
                        if (jj >= nj) break;
                        const int t = tfirst + jj;
                        const int b = qb, ii = qi;
                        if (++qi == a.S) {
                            qi = 0;
                            ++qb;
                        }
                        if (t >= a.Mt || !ok) continue;
                        const int c = h * 64 + j_lo + jj;
                        const float u1 = ystage[p * BIG_YS + c], u2 = ystage[(p + 64) * BIG_YS + c];
                        if (KIND == G_QKV) {
                            const int hd = a.D >> 1;
                            float r1 = u1, r2 = u2;
                            if (rot) {
                                r1 = u1 * cs[jj].x - u2 * cs[jj].y;
                                r2 = u2 * cs[jj].x + u1 * cs[jj].y;
                            }
                            __nv_bfloat16* dst = (sec < a.H) ? a.q + ((size_t)t * a.H + sec) * a.D
                                                             : (sec == a.H ? a.kst : a.vst) + ((size_t)b * a.kv_rows + a.P + ii) * a.D;
                            dst[d] = __float2bfloat16_rn(r1);
                            dst[d + hd] = __float2bfloat16_rn(r2);
                        } else {
                            a.z[(size_t)t * a.F + pair] = __float2bfloat16_rn(gelu_tanh(u1) * u2);
                        }
                    }
                } else {
                    const int f0 = tile * TILE_ROWS, f = f0 + row;
                    if constexpr (S == 1) {
                        // n = h + gamma * y in place of h: accumulator row `row` (feature f), 32 token
                        // columns at a time, into column f of the [token][feature] tile.
#pragma unroll
                        for (int c0 = 0; c0 < 64; c0 += 32) {
                            uint32_t r[2][16];
                            ptx::tmem_ld_x16(lane_base + (uint32_t)(64 * eg + c0), r[0]);
                            ptx::tmem_ld_x16(lane_base + (uint32_t)(64 * eg + c0 + 16), r[1]);
                            ptx::tmem_ld_wait();
#pragma unroll
                            for (int i = 0; i < 32; ++i) {
                                float* hp = ystage + (64 * eg + c0 + i) * BIG_HS + row;
                                *hp = *hp + gam * __uint_as_float(r[i >> 4][i & 15]);
                            }
                        }
                        ptx::tc_fence_before();
                        ptx::mbar_arrive(&acce[buf]);
                    } else {
                        // Split K: accumulator column c (token c of the unit) belongs to rank c / TOK.
                        // Own columns go to this CTA's slot of the receive buffer, the others to the
                        // outgoing slice of their rank ([token][feature], a warp stores 32
                        // consecutive features of one token).
#pragma unroll
                        for (int c0 = 0; c0 < 64; c0 += 32) {
                            uint32_t r[2][16];
                            ptx::tmem_ld_x16(lane_base + (uint32_t)(64 * eg + c0), r[0]);
                            ptx::tmem_ld_x16(lane_base + (uint32_t)(64 * eg + c0 + 16), r[1]);
                            ptx::tmem_ld_wait();
#pragma unroll
                            for (int hh = 0; hh < 2; ++hh) {
                                // 16 columns never straddle two owners (TOK >= 16).
                                const int col0 = 64 * eg + c0 + 16 * hh, q = col0 / TOK;
                                float* dst = (q == rank ? recvb + (size_t)rank * TOK * BIG_NT
                                                        : sendb + (size_t)(q < rank ? q : q - 1) * TOK * BIG_NT) +
                                             (size_t)(col0 % TOK) * BIG_NT + row;
#pragma unroll
                                for (int i = 0; i < 16; ++i) dst[i * BIG_NT] = __uint_as_float(r[hh][i]);
                            }
                        }
                        ptx::tc_fence_before();
                        ptx::mbar_arrive(&acce[buf]);
                        ptx::fence_proxy_async_smem();   // the outgoing slices, for the bulk copies
                        ptx::named_bar_sync(1, BIG_EPI);
                        if (ew == 0) {
                            // Slices of this unit from the S - 1 peers (lane 0), then this CTA's
                            // slices out, lane q to peer q (the copies issue together).
                            if (lane == 0) ptx::mbar_expect_tx(recvf, (uint32_t)((S - 1) * CF::SLICE));
                            if (lane < S && lane != rank) {
                                const int q = lane;
                                const uint32_t own_slot = ptx::smem_u32(recvb + (size_t)rank * TOK * BIG_NT);
                                const uint32_t rbar = ptx::smem_u32(recvf);
                                ptx::bulk_copy_to_cluster(ptx::dsmem_map(own_slot, (uint32_t)q),
                                                          sendb + (size_t)(q < rank ? q : q - 1) * TOK * BIG_NT,
                                                          (uint32_t)CF::SLICE, ptx::dsmem_map(rbar, (uint32_t)q));
                            }
                            if (lane == 0 && !ptx::mbar_wait_bounded(recvf, j & 1, WAIT_LIMIT_NS)) *flag = DEV_TIMEOUT_MMA;
                        }
                        ptx::named_bar_sync(1, BIG_EPI);   // every partial of this CTA's tokens is here
                        // n = h + gamma * (sum of the S partials in rank order) for tokens cc of this
                        // CTA, feature f: a warp reads and writes 32 consecutive features.
                        for (int cc = eg; cc < TOK; cc += 2) {
                            float y = 0.f;
#pragma unroll
                            for (int q = 0; q < S; ++q) y += recvb[(size_t)(q * TOK + cc) * BIG_NT + row];
                            float* hp = ystage + cc * BIG_HS + row;
                            *hp = *hp + gam * y;
                        }
                    }
                    // The next norm's shift in the last row of each of its token tiles (this tile's rows).
                    if (a.xs && xt == 0 && ok && eg == 0 && rank == 0) {
                        const float bn = a.beta_next[f];
                        for (int x = 0; x < xs_tiles(a.Mt); ++x)
                            a.xs[((size_t)x * 64 + 63) * a.W + f] = __float2bfloat16_rn(bn);
                    }
                    ptx::named_bar_sync(1, BIG_EPI);   // the tile's new residual rows are complete
                    // Warp ew writes tokens TOK / 8 ew..: lane l the features 4 l..4 l + 3 of the new
                    // residual (16 bytes) and of the next norm's operand (8 bytes); the token's sum of
                    // squares over the tile's 128 features is lane 0's butterfly total (slot `tile`).
                    // (A timeout flag may be seen by some lanes only: the warp decides together.)
                    const bool okw = __all_sync(0xffffffffu, ok);
#pragma unroll 4
                    for (int k = 0; k < TOK / 8; ++k) {
                        const int c = (TOK / 8) * ew + k, t = tok0 + rank * TOK + c;
                        if (t >= a.Mt || !okw) break;
                        const float4 n = *(const float4*)(ystage + c * BIG_HS + 4 * lane);
                        *(float4*)(a.hres + (size_t)t * a.W + f0 + 4 * lane) = n;
                        if (a.xs) {
                            const uint2 v = make_uint2(pack_bf16x2((1.f + sg4.x) * n.x, (1.f + sg4.y) * n.y),
                                                       pack_bf16x2((1.f + sg4.z) * n.z, (1.f + sg4.w) * n.w));
                            *(uint2*)(a.xs + (size_t)xs_row(t) * a.W + f0 + 4 * lane) = v;
                        }
                        float sq = ((n.x * n.x + n.y * n.y) + n.z * n.z) + n.w * n.w;
#pragma unroll
                        for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
                        if (lane == 0) a.ss_out[(size_t)tile * a.ss_ld + t] = sq;
                    }
                    // Split K: this CTA has summed its receive buffer (every value read is in the
                    // staging tile, published by the barrier above): each peer may overwrite its slot
                    // (and reuse its outgoing slices) for the next unit. One lane per peer.
                    if (S > 1 && ew == 0 && lane < S - 1) {
                        const int q = lane < rank ? lane : lane + 1;
                        ptx::mbar_arrive_cluster_relaxed(ptx::dsmem_map(ptx::smem_u32(pfree), (uint32_t)q));
                    }
                }
                // Every epilogue thread is done with the staging tile (and rinv) of this tile.
                ptx::named_bar_sync(1, BIG_EPI);
            }
        }
    }

    if (tid == 0 && *flag != 0) set_device_error(a.err, *flag);
    ptx::tc_fence_before();
    __syncthreads();
    // Split K: no copy or arrival of a peer is still aimed at this CTA when it exits.
    if (S > 1) ptx::cluster_sync_all();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc(tmem, 2 * BIG_NT);
}
