// Large-M projection kernel for batched denoises (included by tc_path.cu, inside jpi's anonymous
// namespace), used when a launch has enough tokens to fill the GPU without splitting K.
//
// Output tile = one 128-row weight tile x one 128-row operand tile (128 tokens, or for the
// RMSNorm-fed kinds two 64-row tiles of 63 tokens + one beta row) over the whole K range.
// Persistent: one CTA per SM walks the tiles u = blockIdx.x, + gridDim.x, ... (weight tile
// fastest), and its roles overlap consecutive tiles:
//   warp 0  one thread streams (weight block, operand block) pairs by bulk tensor copies into a
//           ring of BIG_STAGES shared-memory stages (full/empty mbarriers), tile after tile;
//   warp 1  one thread issues the tcgen05.mma chain (M = 128, N = 128, K = 16 each) of a tile
//           into one of two TMEM accumulators (tile j into buffer j mod 2, once the epilogue has
//           read tile j - 2 out of it) and releases each stage through tcgen05.commit;
//   warps 2-9  the epilogue, two groups of four warps (group g takes accumulator columns
//           64g..64g+63): one TMEM lane (weight row) per thread copies its half row to a
//           shared fp32 staging tile, hands the TMEM buffer back, then runs the per-kind
//           epilogue (rotary + scatter, GeGLU, gated residual with the next norm's operand and
//           sums of squares) while the MMAs of the next tile run. Row pairs (p, p + 64) meet
//           through the staging tile; residual rows and rotary factors are loaded in chunks of
//           16 columns (each chunk's loads issued together, the next chunk's in flight).
// The next kernel is released once this CTA's last accumulator is complete. All waits are
// bounded.

constexpr int BIG_NT = 128;                       // operand rows per tile
constexpr int BIG_STAGES = 4;
constexpr int BIG_EPI = 256;                     // epilogue threads: two groups of 4 warps
constexpr int BIG_THREADS = 64 + BIG_EPI;
constexpr int BIG_XBYTES = BIG_NT * KBLK * 2;     // 16 KB operand block
constexpr int BIG_STAGE_BYTES = TILE_BYTES + BIG_XBYTES;
constexpr int BIG_YS = BIG_NT + 1;                // fp32 staging row stride: conflict-free rows and columns
constexpr int BIG_YBYTES = TILE_ROWS * BIG_YS * 4;

__host__ __device__ constexpr int big_smem_bytes() {
    // stages | staging tile | rinv[128] | bars (full, empty, acc full[2], acc empty[2]) + TMEM slot + flag
    return BIG_STAGES * BIG_STAGE_BYTES + BIG_YBYTES + BIG_NT * 4 + 128;
}

template <int KIND>
__global__ void __launch_bounds__(BIG_THREADS, 1) k_tc_gemm_big(const __grid_constant__ CUtensorMap wmap,
                                                             const __grid_constant__ CUtensorMap xmap,
                                                             const __grid_constant__ GemmArgs a) {
    constexpr bool NORM_IN = (KIND == G_QKV || KIND == G_GU);
    constexpr int TT = NORM_IN ? 2 * XS_TOKENS : BIG_NT;   // tokens per tile
    constexpr uint32_t IDESC = ptx::idesc_bf16_f32(TILE_ROWS, BIG_NT);

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (ptx::smem_u32(smem_raw) & 1023u)) & 1023u);
    uint8_t* stages = smem;                                             // [stage][W 16 KB | X 16 KB]
    float* ystage = (float*)(smem + BIG_STAGES * BIG_STAGE_BYTES);      // [128][BIG_YS]
    float* rinv_s = (float*)((uint8_t*)ystage + BIG_YBYTES);            // [128]
    uint64_t* full = (uint64_t*)(rinv_s + BIG_NT);
    uint64_t* empty = full + BIG_STAGES;
    uint64_t* accf = empty + BIG_STAGES;   // [2] accumulator buffer holds a finished tile
    uint64_t* acce = accf + 2;             // [2] the epilogue has read it out
    uint32_t* tmem_slot = (uint32_t*)(acce + 2);
    int* flag = (int*)(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int nkb = a.nkb;
    const int ntiles = a.ntiles;
    const int nxt = (a.Mt + TT - 1) / TT;
    const int total = ntiles * nxt;
    const int u0 = blockIdx.x, du = gridDim.x;

    if (warp == 1) {
        ptx::tmem_alloc(tmem_slot, 2 * BIG_NT);
        ptx::tmem_relinquish();
    }
    if (tid == 0) {
        for (int i = 0; i < 2 * BIG_STAGES; ++i) ptx::mbar_init(&full[i], 1);
        ptx::mbar_init(&accf[0], 1);
        ptx::mbar_init(&accf[1], 1);
        ptx::mbar_init(&acce[0], BIG_EPI);
        ptx::mbar_init(&acce[1], BIG_EPI);
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
            auto load_w = [&](int tile, int kb, int s) {
                ptx::mbar_expect_tx(&full[s], (uint32_t)BIG_STAGE_BYTES);
                ptx::tma_load_2d(stages + s * BIG_STAGE_BYTES, &wmap, &full[s], 0, (tile * nkb + kb) * TILE_ROWS, pol);
            };
            ptx::prefetch_tmap(&xmap);
            auto load_x = [&](int xt, int kb, int s) {
                uint8_t* xs = stages + s * BIG_STAGE_BYTES + TILE_BYTES;
                ptx::tma_load_2d(xs, &xmap, &full[s], kb * KBLK, xt * BIG_NT, pol);
                ptx::tma_load_2d(xs + XBLK_BYTES, &xmap, &full[s], kb * KBLK, xt * BIG_NT + NT, pol);
            };
            // Weight blocks of the first tile's first stages do not depend on the previous kernel.
            const int npre = u0 < total ? (nkb < BIG_STAGES ? nkb : BIG_STAGES) : 0;
            for (int kb = 0; kb < npre; ++kb) load_w(u0 % ntiles, kb, kb);
            ptx::grid_dep_wait();
            int it = 0;   // k-block counter over this CTA's tiles: stage it mod STAGES
            bool ok = true;
            for (int u = u0; u < total && ok; u += du) {
                const int tile = u % ntiles, xt = u / ntiles;
                for (int kb = 0; kb < nkb; ++kb, ++it) {
                    const int s = it % BIG_STAGES, n = it / BIG_STAGES;
                    if (it < npre) {   // first tile, weights already in flight
                        load_x(xt, kb, s);
                        continue;
                    }
                    if (it >= BIG_STAGES && !ptx::mbar_wait_bounded(&empty[s], (n - 1) & 1, WAIT_LIMIT_NS)) {
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
                    const int s = it % BIG_STAGES, n = it / BIG_STAGES;
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
        // ---- epilogue: thread et = TMEM lane (weight row) of the accumulator ----
        const int et = (tid - 64) & 127, eg = (tid - 64) >> 7;   // thread within its group, group
        const int row = (warp & 3) * 32 + lane;
        ptx::grid_dep_wait();
        // Pair / token-half of this thread in the norm-fed epilogues.
        const int p = et & 63, h = et >> 6;
        bool ok = true;
        for (int u = u0, j = 0; u < total; u += du, ++j) {
            const int buf = j & 1;
            const int tile = u % ntiles, xt = u / ntiles;
            const int tok0 = xt * TT;
            const int pair = tile * 64 + p;
            int sec = 0, d = 0;
            if (KIND == G_QKV) {
                const int hd = a.D >> 1;
                sec = pair / hd;
                d = pair - sec * hd;
            }
            if (NORM_IN && eg == 0) {
                // Column scale: rinv of the column's token (sums of squares in slot order), 1 for
                // the beta columns 63 and 127.
                const int c = et;
                const int t = tok0 + (c >> 6) * XS_TOKENS + (c & 63);
                float r = 1.f;
                if ((c & 63) != 63) {
                    r = 0.f;
                    if (t < a.Mt) {
                        float s = 0.f;
                        for (int sl = 0; sl < a.nslot; ++sl) s += a.ss[(size_t)sl * a.ss_ld + t];
                        r = rsqrtf(s * a.inv_w + a.eps);
                    }
                }
                rinv_s[c] = r;
            }
            if (!ptx::mbar_wait_bounded(&accf[buf], (j >> 1) & 1, WAIT_LIMIT_NS)) *flag = DEV_TIMEOUT_MMA;
            ptx::named_bar_sync(1, BIG_EPI);   // rinv_s published; every epilogue thread saw the MMAs done
            ptx::tc_fence_after();
            // This CTA's last accumulator is complete: the next kernel may start streaming its weights.
            if (u + du >= total) ptx::grid_dep_launch();
            ok = ok && *flag == 0;

            const uint32_t lane_base = tmem + (uint32_t)(buf * BIG_NT) + ((uint32_t)((warp & 3) * 32) << 16);
            // Accumulator row -> staging row (NORM_IN: y = rinv * acc + W beta of the column's
            // 64-group), then the TMEM buffer goes back to the MMA thread.
            float beta = 0.f;   // W beta of this group's 64 columns (column 64 eg + 63)
            if (NORM_IN) {
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
                        ystage[row * BIG_YS + c] =
                            !NORM_IN ? v : (c & 63) == 63 ? 0.f : rinv_s[c] * v + beta;
                    }
            }
            ptx::tc_fence_before();
            ptx::mbar_arrive(&acce[buf]);

            if (NORM_IN) {
                ptx::named_bar_sync(1, BIG_EPI);   // staging rows of the pair partners written
                // Thread (pair p, column half h): rows p and p + 64 of this tile for 63 tokens, in
                // chunks of 16 tokens whose rotary factors are loaded together.
                const int j_lo = 32 * eg, j_hi = eg ? XS_TOKENS : 32;   // this group's tokens
                const int tfirst = tok0 + h * XS_TOKENS + j_lo;
                int qb = tfirst / a.S, qi = tfirst - qb * a.S;   // request and position of the token
                const bool rot = KIND == G_QKV && a.rope && sec <= a.H;
                // Rotary factors of tokens j0..j0+15, loaded together; position ql advances with j.
                int ql = qi;
                auto load_cs = [&](int j0, float2 (&dst)[16]) {
                    const int hd = a.D >> 1;
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const bool in = rot && j0 + i < j_hi - j_lo && tfirst + j0 + i < a.Mt;
                        dst[i] = in ? __ldg(a.rope + (size_t)(a.P + ql) * hd + d) : make_float2(1.f, 0.f);
                        if (++ql == a.S) ql = 0;
                    }
                };
                float2 cs[16];
                load_cs(0, cs);
                for (int j0 = 0; j0 < j_hi - j_lo; j0 += 16) {
                    float2 cn[16];
                    if (j0 + 16 < j_hi - j_lo) load_cs(j0 + 16, cn);   // the next chunk's factors in flight
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int jj = j0 + i;
                        if (jj >= j_hi - j_lo) break;
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
                                r1 = u1 * cs[i].x - u2 * cs[i].y;
                                r2 = u2 * cs[i].x + u1 * cs[i].y;
                            }
                            __nv_bfloat16* dst = (sec < a.H) ? a.q + ((size_t)t * a.H + sec) * a.D
                                                             : (sec == a.H ? a.kst : a.vst) + ((size_t)b * a.kv_rows + a.P + ii) * a.D;
                            dst[d] = __float2bfloat16_rn(r1);
                            dst[d + hd] = __float2bfloat16_rn(r2);
                        } else {
                            a.z[(size_t)t * a.F + pair] = __float2bfloat16_rn(gelu_tanh(u1) * u2);
                        }
                    }
#pragma unroll
                    for (int i = 0; i < 16; ++i) cs[i] = cn[i];
                }
            } else {
                const int f = tile * TILE_ROWS + row;
                const float g = a.gamma[f];
                const float sn = a.xs ? a.sigma_next[f] : 0.f;
                // 16 columns at a time; the next chunk's residual values are loaded (together)
                // before this chunk is updated, so their latency overlaps the updates.
                float hv[16];
                auto load_h = [&](int c0, float (&dst)[16]) {
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int t = tok0 + c0 + i;
                        dst[i] = t < a.Mt ? a.hres[(size_t)t * a.W + f] : 0.f;
                    }
                };
                const int cb = 64 * eg, ce = cb + 64;   // this group's columns
                load_h(cb, hv);
#pragma unroll 1
                for (int c0 = cb; c0 < ce; c0 += 16) {
                    float hn[16];
                    if (c0 + 16 < ce) load_h(c0 + 16, hn);
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int c = c0 + i, t = tok0 + c;
                        float sq = 0.f;
                        if (t < a.Mt && ok) {
                            const float n = hv[i] + g * ystage[row * BIG_YS + c];
                            a.hres[(size_t)t * a.W + f] = n;
                            if (a.xs) a.xs[(size_t)xs_row(t) * a.W + f] = __float2bfloat16_rn((1.f + sn) * n);
                            sq = n * n;
                        }
                        ystage[row * BIG_YS + c] = sq;
                    }
#pragma unroll
                    for (int i = 0; i < 16; ++i) hv[i] = hn[i];
                }
                // The next norm's shift in the last row of each of its token tiles (this tile's rows).
                if (a.xs && xt == 0 && ok && eg == 0) {
                    const float bn = a.beta_next[f];
                    for (int x = 0; x < xs_tiles(a.Mt); ++x)
                        a.xs[((size_t)x * 64 + 63) * a.W + f] = __float2bfloat16_rn(bn);
                }
                ptx::named_bar_sync(1, BIG_EPI);
                // Sum of squares of token c over this tile's 128 features, in row order: slot `tile`.
                const int c = et, t = tok0 + c;
                if (eg == 0 && t < a.Mt && ok) {
                    float s = 0.f;
                    for (int r = 0; r < TILE_ROWS; ++r) s += ystage[r * BIG_YS + c];
                    a.ss_out[(size_t)tile * a.ss_ld + t] = s;
                }
            }
            // Every epilogue thread is done with the staging tile and rinv_s of this tile.
            ptx::named_bar_sync(1, BIG_EPI);
        }
    }

    if (tid == 0 && *flag != 0) set_device_error(a.err, *flag);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc(tmem, 2 * BIG_NT);
}
