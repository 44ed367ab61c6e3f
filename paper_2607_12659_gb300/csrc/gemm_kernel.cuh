// The tensor-core projection kernel (included by tc_path.cu, inside jpi's anonymous namespace).
//
// One CTA = one (128-row weight tile, K range) unit; the CTAs of a cluster share the tile and
// split its K range. Per 64-token tile:
//   1. B operand: bulk tensor copies of the bf16/fp16 activation blocks; for the RMSNorm-fed
//      projections the norm and the time-conditioned scale/shift are applied in place.
//   2. tcgen05.mma of the weight blocks (loaded before the grid-dependency wait) into TMEM.
//   3. Split-K reduction: each CTA converts its product to an fp16 partial in its own shared
//      memory and at once pushes the rows owned by every other rank of the cluster to that rank
//      with bulk shared::cluster copies (completion counted on the owner's mbarrier, whose
//      initialisation the whole cluster has seen at kernel start); the owner sums the slices in
//      rank order from its own shared memory. The receive buffer is used by nothing else.
//   4. Epilogue on the owned rows. A CTA arrives on the cluster barrier as soon as everything
//      addressed to it has landed and waits on it only before it exits (or, with several token
//      tiles, before the next tile reuses the buffers), so the barrier is off the critical path.
//
// Partial rows are 64 fp16 tokens (128 bytes) with their 16-byte chunks XOR-swizzled by the row
// index mod 8, which keeps both the TMEM write-out (one row per lane) and the reduction reads
// (16 lanes per row) free of bank conflicts without padding.

template <int KIND>
__global__ void __launch_bounds__(GEMM_THREADS, 2) k_tc_gemm(const __grid_constant__ CUtensorMap wmap,
                                                          const __grid_constant__ CUtensorMap xmap,
                                                          const __grid_constant__ GemmArgs a) {
    constexpr bool NORM_IN = (KIND == G_QKV || KIND == G_GU);
    constexpr bool RESID = (KIND == G_O || KIND == G_DOWN);
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
    float* rpart = (float*)(smem + L.misc);                // [4][NT] sums of squares (norm-fed)
    float* sig = rpart + 4 * NT;                           // [kpb * KBLK] this CTA's sigma slice
    float* bet = sig + a.kpb * KBLK;                       // [kpb * KBLK] this CTA's beta slice
    float* ssred = (float*)(smem + L.ssred);               // [2][NT] (residual kinds)
    uint64_t* bars = (uint64_t*)(smem + L.bars);           // weights, X, MMA done, received
    uint32_t* tmem_slot = (uint32_t*)(bars + 4);
    int* flag = (int*)(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int rank = (int)ptx::cluster_rank();
    const int tile = blockIdx.x / a.splits;
    const int kb0 = rank * a.kpb;
    const int npairs = 64 / a.splits, p0 = rank * npairs;
    // Epilogue item = (token quad, owned pair) with the pair fastest, so that consecutive lanes
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
    }
    // The modulation vectors come from the time-conditioning kernels, which precede this launch
    // by at least two kernels; a dependent launch starts only after its predecessor has passed
    // its own dependency wait, so they are complete here and can be read before ours.
    if (NORM_IN) {
        for (int i = tid; i < a.kpb * KBLK; i += GEMM_THREADS) {
            sig[i] = a.sigma[kb0 * KBLK + i];
            bet[i] = a.beta[kb0 * KBLK + i];
        }
    }
    // Every CTA's receive barrier is initialised before any CTA pushes into it: arrive now, wait
    // before the first push (the round trip overlaps the previous kernel and this one's loads).
    ptx::cluster_arrive();
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();

    const int ntt = (a.Mt + NT - 1) / NT;
    for (int tt = 0; tt < ntt; ++tt) {
        const int tok0 = tt * NT;
        const bool last = tt == ntt - 1;
        // ---- 1. B operand ----
        if (tid == 0) {
            const uint64_t pol = ptx::l2_policy_evict_first();
            ptx::mbar_expect_tx(&bars[1], (uint32_t)(a.kpb * XBLK_BYTES));
            for (int j = 0; j < a.kpb; ++j)
                ptx::tma_load_2d(xsm + j * XBLK_BYTES, &xmap, &bars[1], (kb0 + j) * KBLK, tok0, pol);
        }
        if (tid == 32)
            ptx::mbar_expect_tx(&bars[3], (uint32_t)((a.splits - 1) * 2 * npairs * 128));
        if (NORM_IN) {
            // Sum of squares of token t: slots g, g + 4, ... summed by thread (g, t); the four
            // partials are added in order where they are used.
            // The loads of up to 32 slots are issued together, then added in slot order.
            const int t = tid & (NT - 1), g = tid >> 6;
            const int tok = tok0 + t;
            float s = 0.f;
            for (int base = g; base < a.nslot; base += 4 * 32) {
                float v[32];
#pragma unroll
                for (int u = 0; u < 32; ++u) {
                    const int sl = base + 4 * u;
                    v[u] = (tok < a.Mt && sl < a.nslot) ? a.ss[(size_t)sl * a.ss_ld + tok] : 0.f;
                }
#pragma unroll
                for (int u = 0; u < 32; ++u) s += v[u];
            }
            rpart[g * NT + t] = s;
        }
        if (!ptx::mbar_wait_bounded(&bars[1], tt & 1, WAIT_LIMIT_NS)) *flag = DEV_TIMEOUT_WEIGHTS;
        if (NORM_IN) {
            __syncthreads();
            // In place: u = h * rinv * (1 + sigma) + beta on each swizzled 16-byte chunk. Thread
            // = physical chunk q of rows tr and tr + 32 (GEMM_THREADS / 8 == 32); both rows hold
            // the same logical chunk c = q ^ (tr mod 8), so sigma/beta are read once per block.
            static_assert(GEMM_THREADS == 8 * 32 && GEMM_THREADS == 4 * NT, "thread mappings");
            const int q = tid & 7, tr = tid >> 3, c = q ^ (tr & 7);
            auto rinv_of = [&](int t) {
                const float s = ((rpart[t] + rpart[NT + t]) + rpart[2 * NT + t]) + rpart[3 * NT + t];
                return rsqrtf(s * a.inv_w + a.eps);
            };
            const float r0 = (tok0 + tr < a.Mt) ? rinv_of(tr) : 0.f;
            const float r1 = (tok0 + tr + 32 < a.Mt) ? rinv_of(tr + 32) : 0.f;
            for (int j = 0; j < a.kpb; ++j) {
                const int kl = j * KBLK + c * 8;
                uint4* pa = (uint4*)(xsm + j * XBLK_BYTES + tr * 128 + q * 16);
                uint4* pb = pa + 32 * 128 / 16;
                const uint4 v0 = *pa, v1 = *pb;
                const float4 s0 = *(const float4*)(sig + kl), s1 = *(const float4*)(sig + kl + 4);
                const float4 b0 = *(const float4*)(bet + kl), b1 = *(const float4*)(bet + kl + 4);
                const float gm[8] = {1.f + s0.x, 1.f + s0.y, 1.f + s0.z, 1.f + s0.w,
                                     1.f + s1.x, 1.f + s1.y, 1.f + s1.z, 1.f + s1.w};
                const float bb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
                const uint32_t in0[4] = {v0.x, v0.y, v0.z, v0.w}, in1[4] = {v1.x, v1.y, v1.z, v1.w};
                uint32_t o0[4], o1[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float2 h0 = unpack_half2(in0[e]), h1 = unpack_half2(in1[e]);
                    // Padding tokens (>= Mt) become exactly zero: rinv 0 and no shift.
                    o0[e] = r0 != 0.f ? pack_bf16x2(h0.x * r0 * gm[2 * e] + bb[2 * e], h0.y * r0 * gm[2 * e + 1] + bb[2 * e + 1]) : 0u;
                    o1[e] = r1 != 0.f ? pack_bf16x2(h1.x * r1 * gm[2 * e] + bb[2 * e], h1.y * r1 * gm[2 * e + 1] + bb[2 * e + 1]) : 0u;
                }
                *pa = make_uint4(o0[0], o0[1], o0[2], o0[3]);
                *pb = make_uint4(o1[0], o1[1], o1[2], o1[3]);
            }
            ptx::fence_proxy_async_smem();
        }
        __syncthreads();

        // ---- 2. MMA: D[128 rows][NT tokens] over this CTA's K blocks ----
        if (tid == 0 && *flag == 0) {
            if (tt == 0 && !ptx::mbar_wait_bounded(&bars[0], 0, WAIT_LIMIT_NS)) {
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
                ptx::mma_commit(&bars[2]);
            }
        }
        // Epilogue inputs from global memory that do not depend on the product: issued now so
        // their latency overlaps the MMA and the exchange (first item of this thread only).
        float hv1[4] = {0.f, 0.f, 0.f, 0.f}, hv2[4] = {0.f, 0.f, 0.f, 0.f}, g1 = 0.f, g2 = 0.f;
        float2 cs[4] = {make_float2(1.f, 0.f), make_float2(1.f, 0.f), make_float2(1.f, 0.f), make_float2(1.f, 0.f)};
        auto prefetch = [&](int item) {
            const int p = p0 + item % npairs, t0 = (item / npairs) * 4;
            const int f1 = tile * TILE_ROWS + p, f2 = f1 + 64;
            if (RESID) {
                g1 = a.gamma[f1];
                g2 = a.gamma[f2];
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int tok = tok0 + t0 + e;
                hv1[e] = hv2[e] = 0.f;
                cs[e] = make_float2(1.f, 0.f);
                if (tok < a.Mt) {
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
        if (tid < nitems) prefetch(tid);
        if (*flag == 0 && !ptx::mbar_wait_bounded(&bars[2], tt & 1, WAIT_LIMIT_NS)) *flag = DEV_TIMEOUT_MMA;
        __syncthreads();
        const bool ok = *flag == 0;
        ptx::tc_fence_after();

        // ---- 3a. TMEM -> fp16 partial in shared memory (warp w: lanes 32 (w mod 4), half w / 4).
        // fp16 halves the bytes the cluster exchanges; a partial beyond the fp16 range raises a
        // device error instead of overflowing silently.
        if (ok) {
            const int row = (warp & 3) * 32 + lane, cbase = (warp >> 2) * (NT / 2);
            bool range_ok = true;
#pragma unroll
            for (int c0 = 0; c0 < NT / 2; c0 += 16) {
                uint32_t r[16];
                ptx::tmem_ld_x16(tmem + ((uint32_t)((warp & 3) * 32) << 16) + (uint32_t)(cbase + c0), r);
                ptx::tmem_ld_wait();
                uint32_t hp[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const float v0 = __uint_as_float(r[2 * i]), v1 = __uint_as_float(r[2 * i + 1]);
                    range_ok &= fabsf(v0) <= 65000.f && fabsf(v1) <= 65000.f;
                    __half2 hv = __floats2half2_rn(v0, v1);
                    hp[i] = *reinterpret_cast<uint32_t*>(&hv);
                }
                const int ch = (cbase + c0) >> 3;   // logical 16-byte chunk of the first 8 tokens
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
        if (tt == 0) ptx::cluster_wait();   // receive barriers initialised everywhere
        if (tid == 0) {
            const uint32_t chunk = (uint32_t)(npairs * 128);
            const uint32_t bar_u = ptx::smem_u32(&bars[3]);
            for (int r = 0; r < a.splits; ++r) {
                if (r == rank) continue;
                const int slot = rank < r ? rank : rank - 1;   // owner r stores senders != r in order
                const uint32_t dst = ptx::dsmem_map(ptx::smem_u32(recv + (size_t)slot * 2 * npairs * 64), (uint32_t)r);
                const uint32_t rbar = ptx::dsmem_map(bar_u, (uint32_t)r);
                ptx::bulk_copy_to_cluster(dst, part + (size_t)r * npairs * 64, chunk, rbar);
                ptx::bulk_copy_to_cluster(dst + chunk, part + (size_t)(r * npairs + 64) * 64, chunk, rbar);
            }
        }
        if (!ptx::mbar_wait_bounded(&bars[3], tt & 1, WAIT_LIMIT_NS)) *flag = DEV_TIMEOUT_MMA;
        // Everything addressed to this CTA has landed (seen through its own mbarrier); once all
        // ranks arrive, every copy out of this CTA's partial has completed as well. Nothing else
        // is published through this barrier, so the arrival is relaxed.
        if (last) ptx::cluster_arrive_relaxed();

        // ---- 4. rank-ordered sum of the slices (own rows read in place) + epilogue ----
        float ssq[4] = {0.f, 0.f, 0.f, 0.f};
        for (int item = tid; item < nitems; item += GEMM_THREADS) {
            if (item != tid) prefetch(item);
            const int pi = item % npairs, quad = item / npairs, t0 = quad * 4, p = p0 + pi;
            // Offset of tokens t0..t0+3 inside a swizzled row with key p mod 8 (= (p + 64) mod 8).
            const int off = (((quad >> 1) ^ (p & 7)) << 3) + ((quad & 1) << 2);
            float4 y1 = make_float4(0.f, 0.f, 0.f, 0.f), y2 = y1;
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
            }
            if (!ok) continue;
            const int f1 = tile * TILE_ROWS + p, f2 = f1 + 64;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int tok = tok0 + t0 + e;
                if (tok >= a.Mt) continue;
                const float u1 = f4get(y1, e), u2 = f4get(y2, e);
                if (KIND == G_QKV) {
                    const int hd = a.D >> 1, pair = tile * 64 + p;
                    const int sec = pair / hd, d = pair - sec * hd;
                    const int b = tok / a.S, pos = a.P + (tok - b * a.S);
                    float r1 = u1, r2 = u2;
                    if (sec <= a.H) {
                        r1 = u1 * cs[e].x - u2 * cs[e].y;
                        r2 = u2 * cs[e].x + u1 * cs[e].y;
                    }
                    __nv_bfloat16* dst = (sec < a.H) ? a.q + ((size_t)tok * a.H + sec) * a.D
                                                     : (sec == a.H ? a.kst : a.vst) + ((size_t)b * a.kv_rows + pos) * a.D;
                    dst[d] = __float2bfloat16_rn(r1);
                    dst[d + hd] = __float2bfloat16_rn(r2);
                } else if (KIND == G_GU) {
                    a.z[(size_t)tok * a.F + tile * 64 + p] = __float2bfloat16_rn(gelu_tanh(u1) * u2);
                } else {
                    const float n1 = hv1[e] + g1 * u1;
                    const float n2 = hv2[e] + g2 * u2;
                    a.hres[(size_t)tok * a.W + f1] = n1;
                    a.hres[(size_t)tok * a.W + f2] = n2;
                    a.hx[(size_t)tok * a.W + f1] = __float2half_rn(n1);
                    a.hx[(size_t)tok * a.W + f2] = __float2half_rn(n2);
                    if (!(fabsf(n1) <= 65504.f && fabsf(n2) <= 65504.f)) set_device_error(a.err, DEV_FP16_RANGE);
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
            // This CTA's slot (tile, rank) of the per-token sums the next RMSNorm adds up.
            __syncthreads();
            if (tid < NT && ok && tok0 + tid < a.Mt) {
                float s = ssred[tid];
                if (npairs > 32) s += ssred[NT + tid];
                a.ss_out[(size_t)(tile * a.splits + rank) * a.ss_ld + tok0 + tid] = s;
            }
        }
        // Several token tiles: the next tile's pushes and loads reuse every buffer, so all ranks
        // must be done reading them.
        if (!last) ptx::cluster_sync_all();
    }
    // Pairs the last arrival: after the final tile's receive wait, or (no tokens) the one made
    // before the dependency wait.
    ptx::cluster_wait();

    if (tid == 0 && *flag != 0) set_device_error(a.err, *flag);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 0) ptx::tmem_dealloc(tmem, NT);
}
