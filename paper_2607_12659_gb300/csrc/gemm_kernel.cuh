// The tensor-core projection kernel (included by tc_path.cu, inside jpi's anonymous namespace).
//
// One CTA = one (128-row weight tile, K range) unit; the CTAs of a cluster share the tile and
// split its K range. Per token tile:
//   1. B operand: bulk tensor copies of the bf16 activation blocks. For the RMSNorm-fed
//      projections the operand is xs = (1 + sigma) * h packed as 63 tokens + one beta row, so
//      the product's last column is W beta and the per-token 1 / rms(h) scales the others.
//   2. tcgen05.mma of the weight blocks (loaded before the grid-dependency wait) into TMEM.
//   3. Split-K reduction: each CTA converts its product (scaled by rinv for the norm-fed kinds)
//      to an fp16 partial in its own shared memory and at once
//      pushes the rows owned by every other rank of the cluster to that rank with bulk
//      shared::cluster copies (completion counted on the owner's mbarrier, whose initialisation
//      the whole cluster has seen at kernel start); the owner sums the slices in rank order from
//      its own shared memory. The receive buffer is used by nothing else.
//   4. Epilogue on the owned rows. A CTA arrives on the cluster barrier as soon as everything
//      addressed to it has landed and waits on it only before it exits, so the barrier is off
//      the critical path.
// Token tiles are the grid's y dimension: every (weight tile, token tile) pair is its own
// cluster, and all of them run concurrently (repeated weight tiles come from L2).
//
// Partial rows are 64 fp16 columns (128 bytes) with their 16-byte chunks XOR-swizzled by the row
// index mod 8, which keeps both the TMEM write-out (one row per lane) and the reduction reads
// free of bank conflicts without padding.

template <int KIND>
__global__ void __launch_bounds__(GEMM_THREADS, 2) k_tc_gemm(const __grid_constant__ CUtensorMap wmap,
                                                          const __grid_constant__ CUtensorMap xmap,
                                                          const __grid_constant__ GemmArgs a) {
    constexpr bool NORM_IN = (KIND == G_QKV || KIND == G_GU);
    constexpr bool RESID = (KIND == G_O || KIND == G_DOWN);
    constexpr int TT = NORM_IN ? XS_TOKENS : NT;   // tokens per tile (column 63 is beta if NORM_IN)
    constexpr uint32_t IDESC = ptx::idesc_bf16_f32(TILE_ROWS, NT);

    extern __shared__ uint8_t smem_raw[];
    // Offsetting the shared array itself (not a cast through an integer) keeps every access
    // below in the shared state space.
    uint8_t* smem = smem_raw + ((1024u - (ptx::smem_u32(smem_raw) & 1023u)) & 1023u);
    const GemmSmem L = gemm_layout(a.kpb, a.splits, NORM_IN);
    uint8_t* wsm = smem;                                   // kpb weight tiles
    uint8_t* xsm = smem + L.x;                             // X blocks, then the outgoing partial
    __half* part = (__half*)xsm;                           // [128][64] this CTA's product
    __half* recv = (__half*)(smem + L.recv);               // [splits - 1][2 * npairs][64]
    float* rpart = (float*)(smem + L.misc);                // [3][NT] sums of squares (norm-fed)
    float* rinv_s = rpart + 3 * NT;                        // [NT] column scale (norm-fed)
    float* ssred = (float*)(smem + L.ssred);               // [2][NT] (residual kinds)
    uint64_t* bars = (uint64_t*)(smem + L.bars);           // weights, X, MMA done, received
    uint32_t* tmem_slot = (uint32_t*)(bars + 4);
    int* flag = (int*)(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int rank = (int)ptx::cluster_rank();
    const int tile = blockIdx.x / a.splits;
    const int kb0 = rank * a.kpb;
    const int npairs = 64 / a.splits, p0 = rank * npairs;
    // Epilogue item = (column quad, owned pair) with the pair fastest, so that consecutive lanes
    // write consecutive output features of one token.
    const int nitems = npairs * QUADS;

    if (warp == 0) {
        ptx::tmem_alloc(tmem_slot, NT);
        ptx::tmem_relinquish();
    }
    if (tid == 0) {
        for (int i = 0; i < 4; ++i) ptx::mbar_init(&bars[i], 1);
        ptx::fence_mbar_init();
        *flag = 0;
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    // Weight tiles depend on nothing upstream: start streaming them before the dependency wait.
    if (tid == 0) {
        const uint64_t pol = ptx::l2_policy_evict_first();
        ptx::mbar_expect_tx(&bars[0], (uint32_t)(a.kpb * TILE_BYTES));
        for (int j = 0; j < a.kpb; ++j)
            ptx::tma_load_2d(wsm + j * TILE_BYTES, &wmap, &bars[0], 0,
                             (tile * a.nkb + kb0 + j) * TILE_ROWS, pol);
        ptx::prefetch_tmap(&xmap);   // the operand copy right after the dependency wait
    }
    // Epilogue inputs from global memory that do not depend on the product (first item of this
    // thread only). For the first token tile they are read before the dependency wait: the rotary
    // table is constant, the modulation vectors come from kernels that finished long before, and
    // the residual stream h was last written two projections back (the previous norm-fed kernel
    // passed its own dependency wait, so that writer has completed). Global loads still in flight
    // at the TMEM read-out would slow it down.
    float hv1[4] = {0.f, 0.f, 0.f, 0.f}, hv2[4] = {0.f, 0.f, 0.f, 0.f}, g1 = 0.f, g2 = 0.f;
    float sn1 = 0.f, sn2 = 0.f;
    float2 cs[4] = {make_float2(1.f, 0.f), make_float2(1.f, 0.f), make_float2(1.f, 0.f), make_float2(1.f, 0.f)};
    auto prefetch = [&](int item, int tok0) {
        const int p = p0 + item % npairs, t0 = (item / npairs) * 4;
        const int f1 = tile * TILE_ROWS + p, f2 = f1 + 64;
        if (RESID) {
            g1 = a.gamma[f1];
            g2 = a.gamma[f2];
            if (a.xs) {
                sn1 = a.sigma_next[f1];
                sn2 = a.sigma_next[f2];
            }
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int tok = tok0 + t0 + e;
            hv1[e] = hv2[e] = 0.f;
            cs[e] = make_float2(1.f, 0.f);
            if (t0 + e < TT && tok < a.Mt) {
                if (RESID) {
                    hv1[e] = a.hres[(size_t)tok * a.W + f1];
                    hv2[e] = a.hres[(size_t)tok * a.W + f2];
                }
                if (KIND == G_QKV && a.rope) {
                    const int hd = a.D >> 1, pair = tile * 64 + p;
                    const int sec = pair / hd, d = pair - sec * hd;
                    if (sec <= a.H) cs[e] = __ldg(a.rope + (size_t)(a.P + tok % a.S) * hd + d);
                }
            }
        }
    };
    if (tid < nitems) prefetch(tid, (int)blockIdx.y * TT);
    // Every CTA's receive barrier is initialised before any CTA pushes into it: arrive now, wait
    // before the first push (the round trip overlaps the previous kernel and this one's loads).
    // The initialisation is published by fence.mbarrier_init, so the arrival itself is relaxed
    // (a release arrival would also wait for the weight copies in flight).
    ptx::cluster_arrive_relaxed();
    ptx::grid_dep_wait();
    // When the next kernel may start: right away after the output projection, because the next
    // one (gate/up) streams the largest weight set of the layer (2F x W, four times the output
    // projection's) and needs the whole of this kernel to prefetch it; otherwise after the
    // split-K receive (below), so that the next kernel's weight prefetch does not compete with
    // this kernel's operand loads, MMAs and exchange.
    constexpr bool EARLY_TRIGGER = (KIND == G_O);
    if (EARLY_TRIGGER) ptx::grid_dep_launch();

    {
        const int tt = blockIdx.y;   // token tile
        const int tok0 = tt * TT;
        // ---- 1. B operand (64 rows from row tt * 64 of the operand buffer) ----
        if (tid == 0) {
            const uint64_t pol = ptx::l2_policy_evict_first();
            ptx::mbar_expect_tx(&bars[1], (uint32_t)(a.kpb * XBLK_BYTES));
            for (int j = 0; j < a.kpb; ++j)
                ptx::tma_load_2d(xsm + j * XBLK_BYTES, &xmap, &bars[1], (kb0 + j) * KBLK, tt * NT, pol);
        }
        if (tid == 64)
            ptx::mbar_expect_tx(&bars[3], (uint32_t)((a.splits - 1) * 2 * npairs * 128));

        // ---- 2. MMA: D[128 rows][64 columns] over this CTA's K blocks ----
        if (tid == 0 && *flag == 0) {
            bool ok_in = ptx::mbar_wait_bounded(&bars[1], 0, WAIT_LIMIT_NS);
            if (ok_in) ok_in = ptx::mbar_wait_bounded(&bars[0], 0, WAIT_LIMIT_NS);
            if (!ok_in) {
                *flag = DEV_TIMEOUT_WEIGHTS;
            } else {
                ptx::tc_fence_after();
                const uint32_t wbase = ptx::smem_u32(wsm), xbase = ptx::smem_u32(xsm);
                for (int j = 0; j < a.kpb; ++j)
#pragma unroll
                    for (int kk = 0; kk < KBLK / 16; ++kk)
                        ptx::mma_bf16(tmem, ptx::desc_sw128(wbase + j * TILE_BYTES + kk * 32),
                                      ptx::desc_sw128(xbase + j * XBLK_BYTES + kk * 32), IDESC,
                                      (j | kk) != 0);
            }
            // Committed even after a timeout so that the wait below completes.
            ptx::mma_commit(&bars[2]);
        }
        if (NORM_IN && warp >= 2) {
            // Sum of squares of token t: slots g, g + 3, ... summed by thread (g, t) of warps 2..7,
            // the three partials added in order by thread t; the loads of up to 32 slots are
            // issued together. Column 63 carries W beta and is not scaled.
            const int t = tid & (NT - 1), g = (tid >> 6) - 1;
            const int tok = tok0 + t;
            float s = 0.f;
            for (int base = g; base < a.nslot; base += 3 * 32) {
                float v[32];
#pragma unroll
                for (int u = 0; u < 32; ++u) {
                    const int sl = base + 3 * u;
                    v[u] = (t < TT && tok < a.Mt && sl < a.nslot) ? a.ss[(size_t)sl * a.ss_ld + tok] : 0.f;
                }
#pragma unroll
                for (int u = 0; u < 32; ++u) s += v[u];
            }
            rpart[g * NT + t] = s;
            ptx::named_bar_sync(1, GEMM_THREADS - 64);
            if (tid < 64 + NT) {
                const int c = tid - 64;
                float r = 0.f;
                if (c == TT) r = 1.f;
                else if (tok0 + c < a.Mt)
                    r = rsqrtf(((rpart[c] + rpart[NT + c]) + rpart[2 * NT + c]) * a.inv_w + a.eps);
                rinv_s[c] = r;
            }
        }
        if (!ptx::mbar_wait_bounded(&bars[2], 0, WAIT_LIMIT_NS)) *flag = DEV_TIMEOUT_MMA;
        __syncthreads();
        const bool ok = *flag == 0;
        ptx::tc_fence_after();

        // ---- 3a. TMEM -> fp16 partial in shared memory (warp w: lanes 32 (w mod 4), half w / 4).
        // fp16 halves the bytes the cluster exchanges; a partial beyond the fp16 range raises a
        // device error instead of overflowing silently.
        if (ok) {
            const int row = (warp & 3) * 32 + lane, cbase = (warp >> 2) * (NT / 2);
            const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
            bool range_ok = true;
#pragma unroll
            for (int c0 = 0; c0 < NT / 2; c0 += 16) {
                uint32_t r[16];
                ptx::tmem_ld_x16(lane_base + (uint32_t)(cbase + c0), r);
                ptx::tmem_ld_wait();
                uint32_t hp[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    float v0 = __uint_as_float(r[2 * i]), v1 = __uint_as_float(r[2 * i + 1]);
                    if (NORM_IN) {
                        v0 *= rinv_s[cbase + c0 + 2 * i];
                        v1 *= rinv_s[cbase + c0 + 2 * i + 1];
                    }
                    // Only live columns count: tokens of this launch (and the beta column);
                    // columns past the last token hold products of padding rows.
                    const int col = cbase + c0 + 2 * i, tok = (int)blockIdx.y * TT + col;
                    if (col >= TT || tok < a.Mt) range_ok &= fabsf(v0) <= 65000.f;
                    if (col + 1 >= TT || tok + 1 < a.Mt) range_ok &= fabsf(v1) <= 65000.f;
                    __half2 hv = __floats2half2_rn(v0, v1);
                    hp[i] = *reinterpret_cast<uint32_t*>(&hv);
                }
                const int ch = (cbase + c0) >> 3;   // logical 16-byte chunk of the first 8 columns
                uint4* rowp = (uint4*)(part + row * 64);
                rowp[ch ^ (row & 7)] = make_uint4(hp[0], hp[1], hp[2], hp[3]);
                rowp[(ch + 1) ^ (row & 7)] = make_uint4(hp[4], hp[5], hp[6], hp[7]);
            }
            if (!range_ok) set_device_error(a.err, DEV_FP16_RANGE);
        }
        ptx::tc_fence_before();
        ptx::fence_proxy_async_smem();
        __syncthreads();

        // ---- 3b. push each other rank's rows (pairs r*npairs.. and +64) to that rank ----
        ptx::cluster_wait();   // receive barriers initialised everywhere
        // Lane r of warp 0 sends rank r its rows (the copies to all ranks issue together).
        if (warp == 0 && lane < a.splits && lane != rank) {
            const int r = lane;
            const uint32_t chunk = (uint32_t)(npairs * 128);
            const uint32_t bar_u = ptx::smem_u32(&bars[3]);
            const int slot = rank < r ? rank : rank - 1;   // owner r stores senders != r in order
            const uint32_t dst = ptx::dsmem_map(ptx::smem_u32(recv + (size_t)slot * 2 * npairs * 64), (uint32_t)r);
            const uint32_t rbar = ptx::dsmem_map(bar_u, (uint32_t)r);
            ptx::bulk_copy_to_cluster(dst, part + (size_t)r * npairs * 64, chunk, rbar);
            ptx::bulk_copy_to_cluster(dst + chunk, part + (size_t)(r * npairs + 64) * 64, chunk, rbar);
        }
        if (!ptx::mbar_wait_bounded(&bars[3], 0, WAIT_LIMIT_NS)) *flag = DEV_TIMEOUT_MMA;
        // Everything addressed to this CTA has landed (seen through its own mbarrier); once all
        // ranks arrive, every copy out of this CTA's partial has completed as well. Nothing else
        // is published through this barrier, so the arrival is relaxed.
        ptx::cluster_arrive_relaxed();
        if (!EARLY_TRIGGER) ptx::grid_dep_launch();

        // ---- 4. rank-ordered sum of the slices (own rows read in place) + epilogue ----
        float ssq[4] = {0.f, 0.f, 0.f, 0.f};
        for (int item = tid; item < nitems; item += GEMM_THREADS) {
            if (item != tid) prefetch(item, tok0);
            const int pi = item % npairs, quad = item / npairs, t0 = quad * 4, p = p0 + pi;
            // Offsets of columns t0..t0+3 and of column 63 inside a swizzled row with key p mod 8
            // (= (p + 64) mod 8).
            const int off = (((quad >> 1) ^ (p & 7)) << 3) + ((quad & 1) << 2);
            const int off63 = ((7 ^ (p & 7)) << 3) + 7;
            float4 y1 = make_float4(0.f, 0.f, 0.f, 0.f), y2 = y1;
            float b1 = 0.f, b2 = 0.f;
#pragma unroll 4
            for (int r = 0; r < a.splits; ++r) {
                const __half* s1;
                const __half* s2;
                if (r == rank) {
                    s1 = part + (size_t)p * 64;
                    s2 = part + (size_t)(p + 64) * 64;
                } else {
                    const int slot = r < rank ? r : r - 1;
                    s1 = recv + ((size_t)slot * 2 * npairs + pi) * 64;
                    s2 = recv + ((size_t)slot * 2 * npairs + npairs + pi) * 64;
                }
                f4add(y1, half4_to_float4(*(const uint2*)(s1 + off)));
                f4add(y2, half4_to_float4(*(const uint2*)(s2 + off)));
                if (NORM_IN) {
                    b1 += __half2float(s1[off63]);
                    b2 += __half2float(s2[off63]);
                }
            }
            if (!ok) continue;
            const int f1 = tile * TILE_ROWS + p, f2 = f1 + 64;
            // QKV: head section and index of this pair; request b and position i of the item's
            // first token, advanced token by token (no division per token).
            int sec = 0, d = 0, qb = 0, qi = 0;
            if (KIND == G_QKV) {
                const int hd = a.D >> 1, pair = tile * 64 + p;
                sec = pair / hd;
                d = pair - sec * hd;
                qb = (tok0 + t0) / a.S;
                qi = tok0 + t0 - qb * a.S;
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int tok = tok0 + t0 + e;
                const int b = qb, i = qi;   // request and position of token tok (QKV)
                if (KIND == G_QKV && ++qi == a.S) {
                    qi = 0;
                    ++qb;
                }
                if (t0 + e >= TT || tok >= a.Mt) continue;
                const float u1 = f4get(y1, e) + b1, u2 = f4get(y2, e) + b2;
                if (KIND == G_QKV) {
                    const int hd = a.D >> 1;
                    float r1 = u1, r2 = u2;
                    if (sec <= a.H) {
                        r1 = u1 * cs[e].x - u2 * cs[e].y;
                        r2 = u2 * cs[e].x + u1 * cs[e].y;
                    }
                    __nv_bfloat16* dst = (sec < a.H) ? a.q + ((size_t)tok * a.H + sec) * a.D
                                                     : (sec == a.H ? a.kst : a.vst) + ((size_t)b * a.kv_rows + a.P + i) * a.D;
                    dst[d] = __float2bfloat16_rn(r1);
                    dst[d + hd] = __float2bfloat16_rn(r2);
                } else if (KIND == G_GU) {
                    a.z[(size_t)tok * a.F + tile * 64 + p] = __float2bfloat16_rn(gelu_tanh(u1) * u2);
                } else {
                    const float n1 = hv1[e] + g1 * u1;
                    const float n2 = hv2[e] + g2 * u2;
                    a.hres[(size_t)tok * a.W + f1] = n1;
                    a.hres[(size_t)tok * a.W + f2] = n2;
                    if (a.xs) {
                        const size_t xr = (size_t)xs_row(tok) * a.W;
                        a.xs[xr + f1] = __float2bfloat16_rn((1.f + sn1) * n1);
                        a.xs[xr + f2] = __float2bfloat16_rn((1.f + sn2) * n2);
                    }
                    ssq[e] = fmaf(n1, n1, fmaf(n2, n2, ssq[e]));
                }
            }
            if (RESID) {
                // Sum over the pairs of this item's token quad: the w = min(npairs, 32) lanes
                // that share it, in a fixed butterfly order; then one lane per group records it
                // for its 32-pair chunk (two chunks only when npairs = 64).
                const int w = npairs < 32 ? npairs : 32;
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    float v = ssq[e];
                    for (int o = 1; o < w; o <<= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
                    if ((lane & (w - 1)) == 0) ssred[(pi >> 5) * NT + t0 + e] = v;
                    ssq[e] = 0.f;
                }
            }
        }
        if (RESID) {
            // The next norm's shift in the last row of each of its token tiles (owned features).
            if (a.xs && tt == 0 && ok) {
                const int nxt = xs_tiles(a.Mt);
                for (int idx = tid; idx < nxt * 2 * npairs; idx += GEMM_THREADS) {
                    const int j = idx % (2 * npairs), xt = idx / (2 * npairs);
                    const int f = tile * TILE_ROWS + (j < npairs ? p0 + j : 64 + p0 + j - npairs);
                    a.xs[((size_t)xt * 64 + 63) * a.W + f] = __float2bfloat16_rn(a.beta_next[f]);
                }
            }
            // This CTA's slot (tile, rank) of the per-token sums the next RMSNorm adds up.
            __syncthreads();
            if (tid < NT && ok && tok0 + tid < a.Mt) {
                float s = ssred[tid];
                if (npairs > 32) s += ssred[NT + tid];
                a.ss_out[(size_t)(tile * a.splits + rank) * a.ss_ld + tok0 + tid] = s;
            }
        }
    }
    // Pairs the arrival after the receive wait.
    ptx::cluster_wait();

    if (tid == 0 && *flag != 0) set_device_error(a.err, *flag);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 0) ptx::tmem_dealloc(tmem, NT);
}
