// Large-M projection kernel for batched denoises (included by tc_path.cu, inside jpi's anonymous
// namespace), used when a launch has enough tokens to fill the GPU without splitting K.
//
// One CTA = one 128-row weight tile x one 128-row operand tile (128 tokens, or for the
// RMSNorm-fed kinds two 64-row tiles of 63 tokens + one beta row) over the whole K range:
//   warp 0  one thread streams (weight block, operand block) pairs by bulk tensor copies into a
//           ring of BIG_STAGES shared-memory stages (full/empty mbarriers);
//   warp 1  one thread issues the tcgen05.mma chain (M = 128, N = 128, K = 16 each) into one
//           TMEM accumulator and releases each stage through tcgen05.commit;
//   warps 2-5  the epilogue: one TMEM lane (weight row) per thread, then the same per-kind
//           epilogues as the split-K kernel (rotary + scatter, GeGLU, gated residual with the
//           next norm's operand and sums of squares). Row pairs (p, p + 64) meet through a
//           shared fp32 staging tile that reuses the stage ring once the MMAs are done. The
//           accumulator is read and the residual rows / rotary factors are loaded in chunks of
//           16-32 columns (each chunk's loads issued together). Two CTAs share an SM, so one
//           CTA's epilogue overlaps the other's mainloop.
// The next kernel is released once the accumulator is complete. All waits are bounded.

constexpr int BIG_NT = 128;                       // operand rows per tile
constexpr int BIG_STAGES = 3;
constexpr int BIG_THREADS = 192;
constexpr int BIG_XBYTES = BIG_NT * KBLK * 2;     // 16 KB operand block
constexpr int BIG_STAGE_BYTES = TILE_BYTES + BIG_XBYTES;
constexpr int BIG_YS = BIG_NT + 1;                // fp32 staging row stride: conflict-free rows and columns

__host__ __device__ constexpr int big_smem_bytes() {
    // stages | rinv[128] | bars (full, empty, acc) + TMEM slot + flag
    return BIG_STAGES * BIG_STAGE_BYTES + BIG_NT * 4 + 128;
}
static_assert(BIG_NT * BIG_YS * 4 <= BIG_STAGES * BIG_STAGE_BYTES, "staging tile fits in the stage ring");

template <int KIND>
__global__ void __launch_bounds__(BIG_THREADS, 2) k_tc_gemm_big(const __grid_constant__ CUtensorMap wmap,
                                                             const __grid_constant__ CUtensorMap xmap,
                                                             const __grid_constant__ GemmArgs a) {
    constexpr bool NORM_IN = (KIND == G_QKV || KIND == G_GU);
    constexpr bool RESID = (KIND == G_O || KIND == G_DOWN);
    constexpr int TT = NORM_IN ? 2 * XS_TOKENS : BIG_NT;   // tokens per tile
    constexpr uint32_t IDESC = ptx::idesc_bf16_f32(TILE_ROWS, BIG_NT);

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (ptx::smem_u32(smem_raw) & 1023u)) & 1023u);
    uint8_t* stages = smem;                                        // [stage][W 16 KB | X 16 KB]
    float* ystage = (float*)smem;                                  // [128][BIG_YS] after the MMAs
    float* rinv_s = (float*)(smem + BIG_STAGES * BIG_STAGE_BYTES); // [128]
    uint64_t* full = (uint64_t*)(rinv_s + BIG_NT);
    uint64_t* empty = full + BIG_STAGES;
    uint64_t* accb = empty + BIG_STAGES;
    uint32_t* tmem_slot = (uint32_t*)(accb + 1);
    int* flag = (int*)(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int tile = blockIdx.x, xt = blockIdx.y;
    const int tok0 = xt * TT;
    const int nkb = a.nkb;

    if (warp == 1) {
        ptx::tmem_alloc(tmem_slot, BIG_NT);
        ptx::tmem_relinquish();
    }
    if (tid == 0) {
        for (int i = 0; i < 2 * BIG_STAGES + 1; ++i) ptx::mbar_init(&full[i], 1);
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
            auto load_w = [&](int kb, int s) {
                ptx::mbar_expect_tx(&full[s], (uint32_t)BIG_STAGE_BYTES);
                ptx::tma_load_2d(stages + s * BIG_STAGE_BYTES, &wmap, &full[s], 0, (tile * nkb + kb) * TILE_ROWS, pol);
            };
            ptx::prefetch_tmap(&xmap);
            auto load_x = [&](int kb, int s) {
                uint8_t* xs = stages + s * BIG_STAGE_BYTES + TILE_BYTES;
                ptx::tma_load_2d(xs, &xmap, &full[s], kb * KBLK, xt * BIG_NT, pol);
                ptx::tma_load_2d(xs + XBLK_BYTES, &xmap, &full[s], kb * KBLK, xt * BIG_NT + NT, pol);
            };
            // Weight blocks of the first stages do not depend on the previous kernel.
            const int npre = nkb < BIG_STAGES ? nkb : BIG_STAGES;
            for (int kb = 0; kb < npre; ++kb) load_w(kb, kb);
            ptx::grid_dep_wait();
            for (int kb = 0; kb < npre; ++kb) load_x(kb, kb);
            for (int kb = npre; kb < nkb; ++kb) {
                const int s = kb % BIG_STAGES, n = kb / BIG_STAGES;
                if (!ptx::mbar_wait_bounded(&empty[s], (n - 1) & 1, WAIT_LIMIT_NS)) {
                    *flag = DEV_TIMEOUT_WEIGHTS;
                    break;
                }
                load_w(kb, s);
                load_x(kb, s);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t base = ptx::smem_u32(stages);
            for (int kb = 0; kb < nkb; ++kb) {
                const int s = kb % BIG_STAGES, n = kb / BIG_STAGES;
                if (!ptx::mbar_wait_bounded(&full[s], n & 1, WAIT_LIMIT_NS)) {
                    *flag = DEV_TIMEOUT_WEIGHTS;
                    break;
                }
                ptx::tc_fence_after();
                const uint32_t w = base + s * BIG_STAGE_BYTES, x = w + TILE_BYTES;
#pragma unroll
                for (int kk = 0; kk < KBLK / 16; ++kk)
                    ptx::mma_bf16(tmem, ptx::desc_sw128(w + kk * 32), ptx::desc_sw128(x + kk * 32), IDESC,
                                  (kb | kk) != 0);
                ptx::mma_commit(&empty[s]);
            }
            // Committed even after a timeout so that the epilogue wakes up.
            ptx::mma_commit(accb);
        }
    } else {
        // ---- epilogue: thread et = TMEM lane (weight row) of the accumulator ----
        const int et = tid - 64;
        const int row = (warp & 3) * 32 + lane;
        ptx::grid_dep_wait();
        // Pair / token-half of this thread in the norm-fed epilogues, and its head section.
        const int p = et & 63, h = et >> 6;
        const int pair = tile * 64 + p;
        int sec = 0, d = 0;
        if (KIND == G_QKV) {
            const int hd = a.D >> 1;
            sec = pair / hd;
            d = pair - sec * hd;
        }
        if (NORM_IN) {
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
        if (!ptx::mbar_wait_bounded(accb, 0, WAIT_LIMIT_NS)) *flag = DEV_TIMEOUT_MMA;
        ptx::named_bar_sync(1, 128);   // rinv_s published; every epilogue thread saw the MMAs done
        ptx::tc_fence_after();
        // The accumulator is complete: the next kernel may start streaming its weights.
        ptx::grid_dep_launch();
        const bool ok = *flag == 0;

        const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
        if (NORM_IN) {
            // y = rinv * acc + (W beta of the column's 64-group), staged as fp32 rows.
            float beta0, beta1;
            {
                uint32_t r[16];
                ptx::tmem_ld_x16(lane_base + 48u, r);
                ptx::tmem_ld_wait();
                beta0 = __uint_as_float(r[15]);
                ptx::tmem_ld_x16(lane_base + 112u, r);
                ptx::tmem_ld_wait();
                beta1 = __uint_as_float(r[15]);
            }
#pragma unroll
            for (int c0 = 0; c0 < BIG_NT; c0 += 16) {
                uint32_t r[16];
                ptx::tmem_ld_x16(lane_base + (uint32_t)c0, r);
                ptx::tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const int c = c0 + i;
                    ystage[row * BIG_YS + c] =
                        (c & 63) == 63 ? 0.f : rinv_s[c] * __uint_as_float(r[i]) + (c < 64 ? beta0 : beta1);
                }
            }
            ptx::named_bar_sync(1, 128);
            // Thread (pair p, column half h): rows p and p + 64 of this tile for 63 tokens, in
            // chunks of 16 tokens whose rotary factors are loaded together.
            const int tfirst = tok0 + h * XS_TOKENS;
            int qb = tfirst / a.S, qi = tfirst - qb * a.S;   // request and position of the token
            const bool rot = KIND == G_QKV && a.rope && sec <= a.H;
            // Rotary factors of tokens j0..j0+15, loaded together; position ql advances with j.
            int ql = qi;
            auto load_cs = [&](int j0, float2 (&dst)[16]) {
                const int hd = a.D >> 1;
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const bool in = rot && j0 + i < XS_TOKENS && tfirst + j0 + i < a.Mt;
                    dst[i] = in ? __ldg(a.rope + (size_t)(a.P + ql) * hd + d) : make_float2(1.f, 0.f);
                    if (++ql == a.S) ql = 0;
                }
            };
            float2 cs[16];
            load_cs(0, cs);
            for (int j0 = 0; j0 < XS_TOKENS; j0 += 16) {
                float2 cn[16];
                if (j0 + 16 < XS_TOKENS) load_cs(j0 + 16, cn);   // the next chunk's factors in flight
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const int j = j0 + i;
                    if (j >= XS_TOKENS) break;
                    const int t = tfirst + j;
                    const int b = qb, ii = qi;
                    if (++qi == a.S) {
                        qi = 0;
                        ++qb;
                    }
                    if (t >= a.Mt || !ok) continue;
                    const int c = h * 64 + j;
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
            // 16 columns at a time; the next chunk's residual values are loaded (together) before
            // this chunk is updated, so their latency overlaps the updates.
            float hv[16];
            auto load_h = [&](int c0, float (&dst)[16]) {
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const int t = tok0 + c0 + i;
                    dst[i] = t < a.Mt ? a.hres[(size_t)t * a.W + f] : 0.f;
                }
            };
            // The accumulator goes to this thread's staging row first, so no global load is in
            // flight while TMEM is read.
#pragma unroll
            for (int c0 = 0; c0 < BIG_NT; c0 += 16) {
                uint32_t r[16];
                ptx::tmem_ld_x16(lane_base + (uint32_t)c0, r);
                ptx::tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 16; ++i) ystage[row * BIG_YS + c0 + i] = __uint_as_float(r[i]);
            }
            load_h(0, hv);
#pragma unroll 1
            for (int c0 = 0; c0 < BIG_NT; c0 += 16) {
                float hn[16];
                if (c0 + 16 < BIG_NT) load_h(c0 + 16, hn);
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
            if (a.xs && xt == 0 && ok) {
                const float bn = a.beta_next[f];
                for (int x = 0; x < xs_tiles(a.Mt); ++x)
                    a.xs[((size_t)x * 64 + 63) * a.W + f] = __float2bfloat16_rn(bn);
            }
            ptx::named_bar_sync(1, 128);
            // Sum of squares of token c over this tile's 128 features, in row order: slot `tile`.
            const int c = et, t = tok0 + c;
            if (t < a.Mt && ok) {
                float s = 0.f;
                for (int r = 0; r < TILE_ROWS; ++r) s += ystage[r * BIG_YS + c];
                a.ss_out[(size_t)tile * a.ss_ld + t] = s;
            }
        }
    }

    if (tid == 0 && *flag != 0) set_device_error(a.err, *flag);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc(tmem, BIG_NT);
}
