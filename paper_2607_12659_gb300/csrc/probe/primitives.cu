// Costs of the hardware primitives that bound the denoise on this GPU, measured directly (a
// diagnostic executable, not part of the library; `python bench.py --primitives` builds and runs
// it and prints its JSON line).
//
// At batch 1 every expert layer is a chain of five stages that each need all of the previous
// stage's output, so the denoise time is set by what it costs to hand data from one set of SMs to
// another and to run a short chain of tensor-core work, not by HBM. At large batch the
// projections and attention are bound by the rate at which an SM takes operands in. Measured here:
//   handoff_flag_us     one SM releases a flag in global memory, another SM polls it with acquire
//                       loads and answers; half the round trip (several SM pairs, median)
//   handoff_8kb_us      the same with 8 KB written before the flag and read after it
//   grid_barrier_us     all co-resident CTAs arrive on one counter and poll it (one CTA per SM)
//   l2_reduce_us        every CTA adds a 32 KB fp32 partial into L2 with red.add (20 targets)
//   l2_bulk_load_us     one CTA's 8 KB bulk copy of L2-resident data into its shared memory
//   stream_gbs          rate at which one CTA per SM takes data in by bulk copies (4 x 16 KB in
//                       flight), from a 32 MB L2-resident buffer with 1, 8, 38, 76 and 152 CTAs
//                       streaming at once (median per CTA), and from a 1 GB buffer (HBM) with 152;
//                       then with 8 and 12 copies in flight (1 and 152 CTAs, L2); then per-thread
//                       16-byte async copies (cp.async, 256 threads, 4 x 16 KB rounds in flight),
//                       and both at once in one CTA (a bulk-copy thread and 256 cp.async threads);
//                       then clusters of 2 and 4 where every CTA fetches 1/2 or 1/4 of each chunk
//                       with a multicast bulk copy into all CTAs of its cluster (bytes received per
//                       CTA: whole chunks; 12 chunks per epoch, a cluster barrier between epochs,
//                       and the same epochs without multicast as the control)
//   mma_cycles          tcgen05.mma issued back to back by one thread (64 in a row, and 4)
//   dsmem_ring_us       4 KB pushed around a ring of 8 CTAs of a cluster, with a cluster barrier
//   coresident_ctas     CTAs of 200 KB shared memory co-resident per cluster size, and whether a
//                       cooperative launch with clusters of 8 is accepted
// Every wait is bounded by %globaltimer (20 ms) and reported in "errors"; every access stays in
// its allocation. One GPU, a few MB of device memory.

#include <cstdio>
#include <cstdlib>
#include <algorithm>
#include <vector>
#include <cuda_runtime.h>

#include "../ptx.h"

namespace {

namespace ptx = jpi::ptx;

constexpr uint64_t LIMIT_NS = 20ull * 1000 * 1000;
constexpr int BIG_SMEM = 200 * 1024;

__device__ __forceinline__ int ld_acquire(const int* p) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_release(int* p, int v) {
    asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
// Polls until *p >= v; false (and the error word set) after LIMIT_NS.
__device__ bool wait_at_least(const int* p, int v, int* err) {
    const uint64_t t0 = ptx::globaltimer_ns();
    for (uint32_t i = 0;; ++i) {
        if (ld_acquire(p) >= v) return true;
        if ((i & 63) == 0 && ptx::globaltimer_ns() - t0 > LIMIT_NS) {
            atomicExch(err, 1);
            return false;
        }
    }
}

// CTA 0 and CTA `peer` alternate: CTA 0 writes `nfloat` values and releases the flag, the peer
// waits for it, reads the values and releases the answer. out[0] = elapsed ns for `iters` rounds.
__global__ void k_handoff(int* flag, int* ack, int peer, int iters, float* data, int nfloat,
                          unsigned long long* out, int* err) {
    if (blockIdx.x != 0 && blockIdx.x != (unsigned)peer) return;
    __shared__ int ok;
    if (threadIdx.x == 0) ok = 1;
    __syncthreads();
    float acc = 0.f;
    const uint64_t t0 = ptx::globaltimer_ns();
    for (int i = 1; i <= iters && ok; ++i) {
        if (blockIdx.x == 0) {
            for (int k = threadIdx.x; k < nfloat; k += blockDim.x) data[k] = (float)i;
            __syncthreads();
            if (threadIdx.x == 0) {
                __threadfence();
                st_release(flag, i);
                if (!wait_at_least(ack, i, err)) ok = 0;
            }
            __syncthreads();
        } else {
            if (threadIdx.x == 0 && !wait_at_least(flag, i, err)) ok = 0;
            __syncthreads();
            for (int k = threadIdx.x; k < nfloat; k += blockDim.x) acc += __ldcg(&data[k]);
            __syncthreads();
            if (threadIdx.x == 0) st_release(ack, i);
        }
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) out[0] = ptx::globaltimer_ns() - t0;
    if (acc == -1.f) out[1] = 1;   // keeps the reads
}

// All CTAs arrive on `counter` and wait for the whole grid, `iters` times.
__global__ void k_grid_barrier(int* counter, int iters, unsigned long long* out, int* err) {
    const int G = gridDim.x;
    const uint64_t t0 = ptx::globaltimer_ns();
    for (int i = 1; i <= iters; ++i) {
        __syncthreads();
        if (threadIdx.x == 0) {
            __threadfence();
            atomicAdd(counter, 1);
            wait_at_least(counter, i * G, err);
        }
        __syncthreads();
        if (*(volatile int*)err) break;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) out[0] = ptx::globaltimer_ns() - t0;
}

// CTA c adds a 128 x 64 fp32 partial (32 KB) into target (c % ntargets), `reps` times.
__global__ void k_l2_reduce(float* dst, int ntargets, int reps) {
    float* t = dst + (size_t)(blockIdx.x % ntargets) * 8192;
    for (int r = 0; r < reps; ++r)
        for (int k = threadIdx.x * 4; k < 8192; k += blockDim.x * 4)
            asm volatile("red.global.add.v4.f32 [%0], {%1,%2,%3,%4};" ::"l"(t + k), "f"(1.f), "f"(1.f), "f"(1.f),
                         "f"(1.f)
                         : "memory");
}

// One CTA: `reps` bulk copies of 8 KB (L2-resident source) into shared memory, one at a time.
__global__ void k_bulk_load(const uint8_t* src, int reps, unsigned long long* out, int* err) {
    extern __shared__ __align__(128) uint8_t sm[];
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        ptx::mbar_init(&bar, 1);
        ptx::fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        const uint64_t t0 = ptx::globaltimer_ns();
        for (int r = 0; r < reps; ++r) {
            ptx::mbar_expect_tx(&bar, 8192);
            asm volatile(
                "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                    ptx::smem_u32(sm)),
                "l"(src + (size_t)(r % 64) * 8192), "r"(8192), "r"(ptx::smem_u32(&bar))
                : "memory");
            if (!ptx::mbar_wait_bounded(&bar, r & 1, LIMIT_NS)) {
                atomicExch(err, 3);
                break;
            }
        }
        out[0] = ptx::globaltimer_ns() - t0;
    }
}

// One thread per CTA streams `reps` 16 KB bulk copies, NS in flight, from chunks of `src`
// (`nchunks` of them; CTA b starts at chunk b * stride) into an NS-slot ring; out[blockIdx.x] =
// elapsed ns.
template <int NS>
__global__ void k_stream(const uint8_t* src, int nchunks, int stride, int reps, unsigned long long* out,
                         int* err) {
    extern __shared__ __align__(128) uint8_t sm[];
    __shared__ __align__(8) uint64_t bar[NS];
    if (threadIdx.x == 0) {
        for (int i = 0; i < NS; ++i) ptx::mbar_init(&bar[i], 1);
        ptx::fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x != 0) return;
    const uint64_t t0 = ptx::globaltimer_ns();
    bool ok = true;
    for (int r = 0; r < reps && ok; ++r) {
        const int s = r % NS;
        if (r >= NS && !ptx::mbar_wait_bounded(&bar[s], ((r - NS) / NS) & 1, LIMIT_NS)) {
            atomicExch(err, 7);
            ok = false;
            break;
        }
        ptx::mbar_expect_tx(&bar[s], 16384);
        const size_t chunk = ((size_t)blockIdx.x * stride + r) % nchunks;
        asm volatile(
            "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                ptx::smem_u32(sm + s * 16384)),
            "l"(src + chunk * 16384), "r"(16384), "r"(ptx::smem_u32(&bar[s]))
            : "memory");
    }
    // The last copies have landed before the CTA exits.
    for (int r = reps - NS < 0 ? 0 : reps - NS; r < reps; ++r)
        if (!ptx::mbar_wait_bounded(&bar[r % NS], (r / NS) & 1, LIMIT_NS)) atomicExch(err, 8);
    out[blockIdx.x] = ptx::globaltimer_ns() - t0;
}

// Warps 1..8 of the CTA stream `reps` rounds of 16 KB with per-thread 16-byte async copies
// (thread k copies bytes 64 k..64 k + 63 of a round), 4 rounds in flight, into a 64 KB ring at
// sm + ring_off; with `bulk` set, thread 0 meanwhile streams `reps` 16 KB bulk copies into
// sm[0, 64 KB) as k_stream<4> does. out[blockIdx.x] = elapsed ns of the slower of the two.
__global__ void k_stream_lsu(const uint8_t* src, int nchunks, int stride, int reps, int bulk,
                             unsigned long long* out, int* err) {
    extern __shared__ __align__(128) uint8_t sm[];
    __shared__ __align__(8) uint64_t bar[4];
    __shared__ unsigned long long t_end[2];
    if (threadIdx.x == 0) {
        for (int i = 0; i < 4; ++i) ptx::mbar_init(&bar[i], 1);
        ptx::fence_mbar_init();
        t_end[0] = t_end[1] = 0;
    }
    __syncthreads();
    const uint64_t t0 = ptx::globaltimer_ns();
    if (threadIdx.x < 32) {
        if (threadIdx.x == 0 && bulk) {
            bool ok = true;
            for (int r = 0; r < reps && ok; ++r) {
                const int s = r & 3;
                if (r >= 4 && !ptx::mbar_wait_bounded(&bar[s], ((r - 4) >> 2) & 1, LIMIT_NS)) {
                    atomicExch(err, 9);
                    ok = false;
                    break;
                }
                ptx::mbar_expect_tx(&bar[s], 16384);
                const size_t chunk = ((size_t)blockIdx.x * stride + r) % nchunks;
                asm volatile(
                    "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                        ptx::smem_u32(sm + s * 16384)),
                    "l"(src + chunk * 16384), "r"(16384), "r"(ptx::smem_u32(&bar[s]))
                    : "memory");
            }
            for (int r = reps - 4 < 0 ? 0 : reps - 4; r < reps; ++r)
                if (!ptx::mbar_wait_bounded(&bar[r & 3], (r >> 2) & 1, LIMIT_NS)) atomicExch(err, 10);
            t_end[0] = ptx::globaltimer_ns() - t0;
        }
    } else {
        const int k = threadIdx.x - 32;   // 0..255
        uint8_t* ring = sm + 65536;
        for (int r = 0; r < reps; ++r) {
            // Chunks offset from the bulk stream's, so the two do not read the same lines.
            const size_t chunk = ((size_t)blockIdx.x * stride + r + nchunks / 2) % nchunks;
            const uint8_t* g = src + chunk * 16384 + 64 * k;
            const uint32_t d = ptx::smem_u32(ring + (r & 3) * 16384 + 64 * k);
#pragma unroll
            for (int q = 0; q < 4; ++q) ptx::cp_async_16(d + 16 * q, g + 16 * q, true);
            asm volatile("cp.async.commit_group;" ::: "memory");
            asm volatile("cp.async.wait_group 3;" ::: "memory");
        }
        asm volatile("cp.async.wait_group 0;" ::: "memory");
        if (k == 0) t_end[1] = ptx::globaltimer_ns() - t0;
    }
    __syncthreads();
    if (threadIdx.x == 0) out[blockIdx.x] = t_end[0] > t_end[1] ? t_end[0] : t_end[1];
}

// Clusters of CL CTAs (CL = 1: the same protocol without multicast), thread 0 of each, in epochs:
// arm 12 slots of 16 KB (one arrival + 16 KB each), cluster barrier (every CTA of the cluster has
// armed its slots and read the previous epoch's), then piece `rank` (16 KB / CL) of each of the
// epoch's 12 chunks is fetched by a multicast bulk copy into that slot of every CTA of the
// cluster, and each CTA waits for its 12 slots: each CTA receives 192 KB an epoch while fetching
// 1/CL of it. Every wait is bounded; the final cluster barrier keeps each CTA alive until nothing
// can still land in it. out[blockIdx.x] = elapsed ns.
template <int CL>
__global__ void k_stream_mc(const uint8_t* src, int nchunks, int stride, int epochs, unsigned long long* out,
                            int* err) {
    constexpr int NSLOT = 12;
    extern __shared__ __align__(128) uint8_t sm[];
    __shared__ __align__(8) uint64_t full[NSLOT];
    const uint32_t rank = ptx::cluster_rank();
    if (threadIdx.x == 0) {
        for (int i = 0; i < NSLOT; ++i) ptx::mbar_init(&full[i], 1);
        ptx::fence_mbar_init();
    }
    __syncthreads();
    const uint64_t t0 = ptx::globaltimer_ns();
    constexpr uint32_t piece = 16384 / CL;
    const uint16_t mask = (uint16_t)((1u << CL) - 1);
    const size_t cluster_id = blockIdx.x / CL;
    bool ok = true;
    for (int e = 0; e < epochs; ++e) {
        if (threadIdx.x == 0)
            for (int i = 0; i < NSLOT; ++i) ptx::mbar_expect_tx(&full[i], 16384);
        __syncwarp();
        ptx::cluster_arrive();
        ptx::cluster_wait();
        if (threadIdx.x == 0) {
            for (int i = 0; i < NSLOT; ++i) {
                const size_t chunk = (cluster_id * stride + (size_t)e * NSLOT + i) % nchunks;
                if (CL == 1)
                    asm volatile(
                        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                            ptx::smem_u32(sm + i * 16384)),
                        "l"(src + chunk * 16384), "r"(16384), "r"(ptx::smem_u32(&full[i]))
                        : "memory");
                else
                    asm volatile(
                        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.multicast::cluster [%0], "
                        "[%1], %2, [%3], %4;" ::"r"(ptx::smem_u32(sm + i * 16384 + rank * piece)),
                        "l"(src + chunk * 16384 + rank * piece), "r"(piece), "r"(ptx::smem_u32(&full[i])), "h"(mask)
                        : "memory");
            }
            for (int i = 0; i < NSLOT; ++i)
                if (ok && !ptx::mbar_wait_bounded(&full[i], e & 1, LIMIT_NS)) {
                    atomicExch(err, 11);
                    ok = false;
                }
        }
        __syncwarp();
    }
    if (threadIdx.x == 0) out[blockIdx.x] = ptx::globaltimer_ns() - t0;
    __syncwarp();
    ptx::cluster_arrive();
    ptx::cluster_wait();
}

// One thread issues `nmma` tcgen05.mma of 128 x N x 16 (bf16, fp32 accumulate) back to back.
// out[0] = cycles to issue them, out[1] = cycles until their commit has arrived.
template <int N>
__global__ void k_mma_issue(int nmma, unsigned long long* out, int* err) {
    extern __shared__ __align__(1024) uint8_t smraw[];
    uint8_t* sm = smraw + ((1024u - (ptx::smem_u32(smraw) & 1023u)) & 1023u);
    __shared__ uint32_t tslot;
    __shared__ __align__(8) uint64_t bar;
    uint8_t* A = sm;           // 128 x 64 bf16
    uint8_t* B = sm + 16384;   // N x 64 bf16
    for (int k = threadIdx.x; k < (16384 + N * 128) / 4; k += blockDim.x) ((uint32_t*)sm)[k] = 0x3c003c00u;
    ptx::fence_proxy_async_smem();
    if (threadIdx.x < 32) {
        ptx::tmem_alloc(&tslot, N);
        ptx::tmem_relinquish();
    }
    if (threadIdx.x == 0) {
        ptx::mbar_init(&bar, 1);
        ptx::fence_mbar_init();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tm = tslot;
    if (threadIdx.x == 0) {
        constexpr uint32_t IDESC = ptx::idesc_bf16_f32(128, N);
        const uint32_t a0 = ptx::smem_u32(A), b0 = ptx::smem_u32(B);
        uint64_t ad[4], bd[4];
        for (int kk = 0; kk < 4; ++kk) {
            ad[kk] = ptx::desc_sw128(a0 + kk * 32);
            bd[kk] = ptx::desc_sw128(b0 + kk * 32);
        }
        const long long c0 = clock64();
        for (int i = 0; i < nmma; ++i) ptx::mma_bf16(tm, ad[i & 3], bd[i & 3], IDESC, i > 0);
        const long long c1 = clock64();
        ptx::mma_commit(&bar);
        if (!ptx::mbar_wait_bounded(&bar, 0, LIMIT_NS)) atomicExch(err, 2);
        const long long c2 = clock64();
        out[0] = (unsigned long long)(c1 - c0);
        out[1] = (unsigned long long)(c2 - c0);
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (threadIdx.x < 32) ptx::tmem_dealloc(tm, N);
}

// A cluster of 8: every rank pushes 4 KB into the next rank's shared memory (completion on that
// rank's mbarrier) and waits for the push it receives, `reps` rounds, each after a cluster barrier.
__global__ void k_dsmem_ring(int reps, unsigned long long* out, int* err) {
    extern __shared__ __align__(128) uint8_t sm[];
    __shared__ __align__(8) uint64_t bar;
    const uint32_t rank = ptx::cluster_rank(), n = 8;
    if (threadIdx.x == 0) {
        ptx::mbar_init(&bar, 1);
        ptx::fence_mbar_init();
    }
    __syncthreads();
    ptx::cluster_sync_all();
    const uint64_t t0 = ptx::globaltimer_ns();
    for (int r = 0; r < reps; ++r) {
        if (threadIdx.x == 0) ptx::mbar_expect_tx(&bar, 4096);
        __syncthreads();
        ptx::cluster_sync_all();   // every rank's receive is armed before anyone pushes
        if (threadIdx.x == 0) {
            const uint32_t dst = ptx::dsmem_map(ptx::smem_u32(sm + 8192), (rank + 1) % n);
            const uint32_t rb = ptx::dsmem_map(ptx::smem_u32(&bar), (rank + 1) % n);
            ptx::bulk_copy_to_cluster(dst, sm, 4096, rb);
            if (!ptx::mbar_wait_bounded(&bar, r & 1, LIMIT_NS)) atomicExch(err, 4);
        }
        __syncthreads();
    }
    ptx::cluster_sync_all();
    if (threadIdx.x == 0 && blockIdx.x == 0) out[0] = ptx::globaltimer_ns() - t0;
}

// Every CTA arrives on the counter and waits for the whole grid (a co-residency check).
__global__ void k_all_resident(int* counter, int* err) {
    if (threadIdx.x == 0) {
        atomicAdd(counter, 1);
        wait_at_least(counter, (int)gridDim.x, err);
    }
}

}  // namespace

#define CK(x)                                                                                       \
    do {                                                                                            \
        cudaError_t e_ = (x);                                                                       \
        if (e_ != cudaSuccess) {                                                                    \
            printf("{\"error\": \"%s: %s\"}\n", #x, cudaGetErrorString(e_));                        \
            return 1;                                                                               \
        }                                                                                           \
    } while (0)

static double median(std::vector<double> v) {
    std::sort(v.begin(), v.end());
    return v[v.size() / 2];
}

int main() {
    CK(cudaSetDevice(0));
    int sms = 0;
    CK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, 0));
    int *d_int = nullptr, *d_err = nullptr;
    unsigned long long* d_out = nullptr;
    float* d_data = nullptr;
    CK(cudaMalloc(&d_int, 4096));
    CK(cudaMalloc(&d_err, 64));
    CK(cudaMalloc(&d_out, 64 * 8 * 4));
    CK(cudaMalloc(&d_data, 4 << 20));
    CK(cudaMemset(d_err, 0, 64));
    CK(cudaMemset(d_data, 0, 4 << 20));
    unsigned long long h[2];

    // Hand-offs between SMs: a cooperative grid of one CTA per SM (200 KB of shared memory each),
    // CTA 0 against several peers.
    CK(cudaFuncSetAttribute(k_handoff, cudaFuncAttributeMaxDynamicSharedMemorySize, BIG_SMEM));
    std::vector<double> flag_us, data_us;
    const int iters = 200;
    for (int nfloat : {0, 2048}) {
        for (int peer : {1, 2, sms / 4, sms / 2, sms - 1}) {
            CK(cudaMemset(d_int, 0, 4096));
            int* flag = d_int;
            int* ack = d_int + 64;
            int pr = peer, it = iters, nf = nfloat;
            void* args[] = {&flag, &ack, &pr, &it, &d_data, &nf, &d_out, &d_err};
            CK(cudaLaunchCooperativeKernel((void*)k_handoff, dim3(sms), dim3(256), args, BIG_SMEM, 0));
            CK(cudaDeviceSynchronize());
            CK(cudaMemcpy(h, d_out, 8, cudaMemcpyDeviceToHost));
            (nfloat ? data_us : flag_us).push_back(h[0] / 1e3 / iters / 2);
        }
    }

    // Grid barrier over one CTA per SM.
    CK(cudaFuncSetAttribute(k_grid_barrier, cudaFuncAttributeMaxDynamicSharedMemorySize, BIG_SMEM));
    CK(cudaMemset(d_int, 0, 4096));
    {
        int it = 200;
        void* args[] = {&d_int, &it, &d_out, &d_err};
        CK(cudaLaunchCooperativeKernel((void*)k_grid_barrier, dim3(sms), dim3(256), args, BIG_SMEM, 0));
        CK(cudaDeviceSynchronize());
        CK(cudaMemcpy(h, d_out, 8, cudaMemcpyDeviceToHost));
    }
    const double barrier_us = h[0] / 1e3 / 200;

    // Split-K style reduction into L2: every SM's CTA adds 32 KB into one of 20 targets.
    cudaEvent_t e0, e1;
    CK(cudaEventCreate(&e0));
    CK(cudaEventCreate(&e1));
    k_l2_reduce<<<sms, 256>>>(d_data, 20, 2);
    CK(cudaDeviceSynchronize());
    CK(cudaEventRecord(e0));
    k_l2_reduce<<<sms, 256>>>(d_data, 20, 20);
    CK(cudaEventRecord(e1));
    CK(cudaEventSynchronize(e1));
    float ms = 0.f;
    CK(cudaEventElapsedTime(&ms, e0, e1));
    const double reduce_us = ms * 1e3 / 20;

    // Bulk copy of 8 KB of L2-resident data, one CTA.
    CK(cudaFuncSetAttribute(k_bulk_load, cudaFuncAttributeMaxDynamicSharedMemorySize, 16384));
    k_bulk_load<<<1, 32, 16384>>>((const uint8_t*)d_data, 64, d_out, d_err);
    CK(cudaDeviceSynchronize());
    k_bulk_load<<<1, 32, 16384>>>((const uint8_t*)d_data, 256, d_out, d_err);
    CK(cudaDeviceSynchronize());
    CK(cudaMemcpy(h, d_out, 8, cudaMemcpyDeviceToHost));
    const double load_us = h[0] / 1e3 / 256;

    // Streaming intake per SM: one CTA per SM (120 KB of shared memory requested, 64 KB used).
    double stream_gbs[5], hbm_gbs = 0.0, deep_gbs[4] = {0.0, 0.0, 0.0, 0.0}, lsu_gbs[4] = {0.0, 0.0, 0.0, 0.0};
    double mc_gbs[4] = {0.0, 0.0, 0.0, 0.0};
    const int nstream[5] = {1, 8, 38, 76, 152};
    {
        uint8_t* d_l2 = nullptr;
        uint8_t* d_hbm = nullptr;
        const size_t l2_bytes = 32u << 20, hbm_bytes = 1ull << 30;
        CK(cudaMalloc(&d_l2, l2_bytes));
        CK(cudaMalloc(&d_hbm, hbm_bytes));
        CK(cudaMemset(d_l2, 1, l2_bytes));
        CK(cudaMemset(d_hbm, 1, hbm_bytes));
        const int smem = 200 * 1024;   // one CTA per SM; 12 slots of 16 KB at most
        CK(cudaFuncSetAttribute(k_stream<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
        CK(cudaFuncSetAttribute(k_stream<8>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
        CK(cudaFuncSetAttribute(k_stream<12>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
        std::vector<unsigned long long> t(sms);
        auto run = [&](auto kern, const uint8_t* src, size_t bytes, int ctas, int stride, int reps) -> double {
            for (int rep = 0; rep < 2; ++rep) {
                kern<<<ctas, 32, smem>>>(src, (int)(bytes / 16384), stride, reps, d_out, d_err);
                if (cudaDeviceSynchronize() != cudaSuccess) return -1.0;
            }
            if (cudaMemcpy(t.data(), d_out, 8 * ctas, cudaMemcpyDeviceToHost) != cudaSuccess) return -1.0;
            std::vector<double> gbs;
            for (int c = 0; c < ctas; ++c) gbs.push_back((double)reps * 16384 / (double)t[c]);
            return median(gbs);
        };
        // L2: every CTA walks the whole 32 MB buffer from its own offset (resident after the
        // first run); HBM: disjoint windows of 400 chunks (6.5 MB) of the 1 GB buffer per CTA.
        for (int i = 0; i < 5; ++i)
            stream_gbs[i] = nstream[i] <= sms ? run(k_stream<4>, d_l2, l2_bytes, nstream[i], 131, 2048) : 0.0;
        hbm_gbs = run(k_stream<4>, d_hbm, hbm_bytes, sms, (int)(hbm_bytes / 16384 / sms), 400);
        deep_gbs[0] = run(k_stream<8>, d_l2, l2_bytes, 1, 131, 2048);
        deep_gbs[1] = run(k_stream<8>, d_l2, l2_bytes, sms, 131, 2048);
        deep_gbs[2] = run(k_stream<12>, d_l2, l2_bytes, 1, 131, 2048);
        deep_gbs[3] = run(k_stream<12>, d_l2, l2_bytes, sms, 131, 2048);
        CK(cudaFuncSetAttribute(k_stream_lsu, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
        // Bytes per CTA: 16 KB per round for cp.async, plus 16 KB per copy for the bulk stream.
        auto run_lsu = [&](int ctas, int bulk) -> double {
            const int reps = 2048;
            for (int rep = 0; rep < 2; ++rep) {
                k_stream_lsu<<<ctas, 288, smem>>>(d_l2, (int)(l2_bytes / 16384), 131, reps, bulk, d_out, d_err);
                if (cudaDeviceSynchronize() != cudaSuccess) return -1.0;
            }
            if (cudaMemcpy(t.data(), d_out, 8 * ctas, cudaMemcpyDeviceToHost) != cudaSuccess) return -1.0;
            std::vector<double> gbs;
            for (int c = 0; c < ctas; ++c) gbs.push_back((double)reps * 16384 * (bulk ? 2 : 1) / (double)t[c]);
            return median(gbs);
        };
        lsu_gbs[0] = run_lsu(1, 0);
        lsu_gbs[1] = run_lsu(sms, 0);
        lsu_gbs[2] = run_lsu(1, 1);
        lsu_gbs[3] = run_lsu(sms, 1);
        // Multicast within clusters of 2 and 4 (and the same protocol in clusters of 1): bytes
        // received per CTA, 192 KB an epoch.
        auto run_mc = [&](auto kern, int cl, int ctas) -> double {
            CK(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(ctas);
            cfg.blockDim = dim3(32);
            cfg.dynamicSmemBytes = smem;
            cudaLaunchAttribute at;
            at.id = cudaLaunchAttributeClusterDimension;
            at.val.clusterDim.x = cl;
            at.val.clusterDim.y = 1;
            at.val.clusterDim.z = 1;
            cfg.attrs = &at;
            cfg.numAttrs = 1;
            const int epochs = 170;   // 2040 chunks of 16 KB per CTA
            for (int rep = 0; rep < 2; ++rep) {
                if (cudaLaunchKernelEx(&cfg, kern, (const uint8_t*)d_l2, (int)(l2_bytes / 16384), 131, epochs, d_out,
                                       d_err) != cudaSuccess)
                    return -1.0;
                if (cudaDeviceSynchronize() != cudaSuccess) return -1.0;
            }
            if (cudaMemcpy(t.data(), d_out, 8 * ctas, cudaMemcpyDeviceToHost) != cudaSuccess) return -1.0;
            std::vector<double> gbs;
            for (int c = 0; c < ctas; ++c) gbs.push_back((double)epochs * 12 * 16384 / (double)t[c]);
            return median(gbs);
        };
        mc_gbs[0] = run_mc(k_stream_mc<1>, 1, 152);
        mc_gbs[1] = run_mc(k_stream_mc<2>, 2, 152);
        mc_gbs[2] = run_mc(k_stream_mc<4>, 4, 144);
        mc_gbs[3] = run_mc(k_stream_mc<2>, 2, 2);
        CK(cudaFree(d_l2));
        CK(cudaFree(d_hbm));
    }

    // tcgen05.mma issue (the second of two runs, so the code is warm).
    double mma[4];
    auto mma_run = [&](auto kern, int n, int count, int slot) -> int {
        const int smem = 16384 + n * 128 + 2048;
        CK(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
        for (int rep = 0; rep < 2; ++rep) {
            kern<<<1, 128, smem>>>(count, d_out, d_err);
            CK(cudaDeviceSynchronize());
        }
        CK(cudaMemcpy(h, d_out, 16, cudaMemcpyDeviceToHost));
        mma[slot] = (double)h[0] / count;
        return 0;
    };
    if (mma_run(k_mma_issue<64>, 64, 64, 0) || mma_run(k_mma_issue<64>, 64, 4, 1) ||
        mma_run(k_mma_issue<128>, 128, 64, 2) || mma_run(k_mma_issue<256>, 256, 64, 3))
        return 1;

    // Distributed shared memory ring in a cluster of 8.
    double ring_us = 0.0;
    {
        CK(cudaFuncSetAttribute(k_dsmem_ring, cudaFuncAttributeMaxDynamicSharedMemorySize, 16384));
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(8);
        cfg.blockDim = dim3(128);
        cfg.dynamicSmemBytes = 16384;
        cudaLaunchAttribute at;
        at.id = cudaLaunchAttributeClusterDimension;
        at.val.clusterDim.x = 8;
        at.val.clusterDim.y = 1;
        at.val.clusterDim.z = 1;
        cfg.attrs = &at;
        cfg.numAttrs = 1;
        int reps = 200;
        CK(cudaLaunchKernelEx(&cfg, k_dsmem_ring, reps, d_out, d_err));
        CK(cudaDeviceSynchronize());
        CK(cudaMemcpy(h, d_out, 8, cudaMemcpyDeviceToHost));
        ring_us = h[0] / 1e3 / reps;
    }

    // Co-resident CTAs at 200 KB of shared memory per cluster size, and a cooperative launch with
    // clusters of 8 over all of them.
    int coresident[5] = {0, 0, 0, 0, 0};
    const int sizes[5] = {1, 2, 4, 8, 16};
    int coop8 = 0;
    CK(cudaFuncSetAttribute(k_all_resident, cudaFuncAttributeMaxDynamicSharedMemorySize, BIG_SMEM));
    if (cudaFuncSetAttribute(k_all_resident, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess)
        cudaGetLastError();
    for (int i = 0; i < 5; ++i) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(sizes[i] * 64);
        cfg.blockDim = dim3(128);
        cfg.dynamicSmemBytes = BIG_SMEM;
        cudaLaunchAttribute at[2];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = sizes[i];
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        int nclusters = 0;
        if (cudaOccupancyMaxActiveClusters(&nclusters, k_all_resident, &cfg) != cudaSuccess) {
            cudaGetLastError();
            nclusters = 0;
        }
        coresident[i] = nclusters * sizes[i];
        if (sizes[i] == 8 && nclusters > 0) {
            CK(cudaMemset(d_int, 0, 4096));
            cfg.gridDim = dim3(nclusters * 8);
            at[1].id = cudaLaunchAttributeCooperative;
            at[1].val.cooperative = 1;
            cfg.numAttrs = 2;
            const cudaError_t e = cudaLaunchKernelEx(&cfg, k_all_resident, d_int, d_err);
            coop8 = (e == cudaSuccess && cudaDeviceSynchronize() == cudaSuccess) ? 1 : 0;
            cudaGetLastError();
        }
    }

    int errs = 0;
    CK(cudaMemcpy(&errs, d_err, 4, cudaMemcpyDeviceToHost));
    printf("{\"sms\": %d, \"handoff_flag_us\": %.3f, \"handoff_flag_us_range\": [%.3f, %.3f], "
           "\"handoff_8kb_us\": %.3f, \"handoff_8kb_us_range\": [%.3f, %.3f], \"grid_barrier_us\": %.3f, "
           "\"l2_reduce_us\": %.3f, \"l2_reduce_bytes\": %d, \"l2_bulk_load_us\": %.3f, "
           "\"mma_cycles\": {\"128x64x16\": %.1f, \"128x64x16_run_of_4\": %.1f, \"128x128x16\": %.1f, "
           "\"128x256x16\": %.1f}, \"dsmem_ring_us\": %.3f, "
           "\"coresident_ctas_200kb\": {\"1\": %d, \"2\": %d, \"4\": %d, \"8\": %d, \"16\": %d}, "
           "\"cooperative_clusters_of_8\": %s, \"stream_gbs_per_cta\": {\"l2_1\": %.1f, \"l2_8\": %.1f, "
           "\"l2_38\": %.1f, \"l2_76\": %.1f, \"l2_152\": %.1f, \"hbm_152\": %.1f, \"l2_1_depth8\": %.1f, "
           "\"l2_152_depth8\": %.1f, \"l2_1_depth12\": %.1f, \"l2_152_depth12\": %.1f, \"l2_1_cp_async\": %.1f, "
           "\"l2_152_cp_async\": %.1f, \"l2_1_bulk_plus_cp_async\": %.1f, \"l2_152_bulk_plus_cp_async\": %.1f, "
           "\"l2_epochs_cluster1_x152\": %.1f, \"l2_multicast_cluster2_x76\": %.1f, "
           "\"l2_multicast_cluster4_x36\": %.1f, \"l2_multicast_cluster2_x1\": %.1f}, \"errors\": %d}\n",
           sms, median(flag_us), *std::min_element(flag_us.begin(), flag_us.end()),
           *std::max_element(flag_us.begin(), flag_us.end()), median(data_us),
           *std::min_element(data_us.begin(), data_us.end()), *std::max_element(data_us.begin(), data_us.end()),
           barrier_us, reduce_us, sms * 32768, load_us, mma[0], mma[1], mma[2], mma[3], ring_us, coresident[0],
           coresident[1], coresident[2], coresident[3], coresident[4], coop8 ? "true" : "false", stream_gbs[0],
           stream_gbs[1], stream_gbs[2], stream_gbs[3], stream_gbs[4], hbm_gbs, deep_gbs[0], deep_gbs[1], deep_gbs[2],
           deep_gbs[3], lsu_gbs[0], lsu_gbs[1], lsu_gbs[2], lsu_gbs[3], mc_gbs[0], mc_gbs[1], mc_gbs[2], mc_gbs[3],
           errs);
    return 0;
}
