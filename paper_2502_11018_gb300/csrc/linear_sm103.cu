// gv_linear / gv_rmsnorm: the target model's projections and norms around the
// tree attention (the decoder layer of the verify forward, GRIFFIN Section 3),
// bf16 on sm_103a.
//
// The projections of a verify step are skinny: the R = B * N <= 256 tree
// nodes times a weight W[N][K] that is read once from HBM (4096 x 4096 up to
// 28672 x 4096 per matrix), so the kernel is a weight stream.  The weight
// rows go on the MMA's M side (tiles of 128 or 256 rows) and the node rows on
// its N side, so a k-block moves 16-32 KB of weights and only 8 KB of node
// rows (64 rows).  TMA fills a ring of shared-memory stages, one lane issues
// tcgen05.mma into a double-buffered TMEM accumulator, and four epilogue warps
// write the tile's fp32 sums (TMEM lane = output column, column = node row).
// A work unit is (weight tile, K split); the split count and tile height are
// chosen so that the units fill the SMs in as few waves as possible, and the
// fp32 partial sums of every split go to the workspace.  gemm_reduce_kernel then
// adds the splits and applies the epilogue (store, residual add, or SwiGLU
// over the gate and up halves), writing bf16.
#include <map>
#include <mutex>
#include <utility>

#include "gv_internal.cuh"
#include "sm103.cuh"

namespace gv {
using namespace sm103;

int make_map_2d(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows,
                uint64_t row_stride_bytes);

constexpr int GM_THREADS = 192;
constexpr int GM_W_TILE = 128 * 128;    // 128 weight rows x 64 bf16

// acc[0..8) += the eight bf16 values at p (16-byte aligned).
__device__ __forceinline__ void bf16x8_add(float* acc, const __nv_bfloat16* p) {
    const uint4 v = *reinterpret_cast<const uint4*>(p);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        acc[2 * e] += __uint_as_float(w[e] << 16);
        acc[2 * e + 1] += __uint_as_float(w[e] & 0xffff0000u);
    }
}

// Column split of the stored output: columns [0, n0) go to out0[rows][n0],
// [n0, n0 + n1) to out1[rows][n1], the rest to out2 (the fused Q/K/V
// projection); n1 == 0 stores everything to out0.
struct OutSplit {
    __nv_bfloat16* out0;
    __nv_bfloat16* out1;
    __nv_bfloat16* out2;
    int n0, n1;
};

// The weight rows are the MMA's M side (tiles of BM = 128 * mm rows, mm MMAs
// per k-step sharing one node-row operand) and the node rows its N side
// (npad = rows rounded up to 32): the big dimension streams, the node rows
// ride along (8 KB per k-block for 64 rows).
struct GemmArgs {
    int rows, npad;          // node rows, MMA N
    int N, K;                // weight rows (GEMM output columns), inner size
    int mm;                  // 128-row MMAs per weight tile
    int n_tiles, KS, kblocks, units;
    int stages, stage_bytes;
    uint32_t tmem_cols;
    int kb_split;            // k-blocks [0, kb_split) from tmap_x, the rest from tmap_x2
    float* part;             // [KS][rows][N] fp32 (split-K through global memory)
    // cluster split-K: the KS CTAs of a tile form a cluster and reduce through
    // distributed shared memory, applying the epilogue themselves
    int n_out, epi;
    const __nv_bfloat16* bias;
    const __nv_bfloat16* residual;
    OutSplit os;
};

// ---- thread-block cluster helpers (distributed shared memory) ----------------
__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
// the address of the same shared-memory location in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t dsmem_addr(uint32_t local, uint32_t rank) {
    uint32_t d;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(d) : "r"(local), "r"(rank));
    return d;
}
__device__ __forceinline__ float4 ld_dsmem_f4(uint32_t addr) {
    float4 v;
    asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(addr)
                 : "memory");
    return v;
}
__device__ __forceinline__ int ld_dsmem_s32(uint32_t addr) {
    int v;
    asm volatile("ld.shared::cluster.s32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
    return v;
}
// every thread of every CTA of the cluster (called convergently by all threads)
__device__ __forceinline__ void cluster_sync_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

template <bool CSK>
__global__ void __launch_bounds__(GM_THREADS, 1)
gemm_tc_kernel(const __grid_constant__ CUtensorMap tmap_x, const __grid_constant__ CUtensorMap tmap_x2,
               const __grid_constant__ CUtensorMap tmap_w, GemmArgs a) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* stage_base = smem_raw;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem_raw + (size_t)a.stages * a.stage_bytes);
    uint64_t* full = bars;
    uint64_t* empty = bars + a.stages;
    uint64_t* tfull = empty + a.stages;
    uint64_t* tempty = tfull + 2;
    uint64_t* drain = tempty + 2;
    uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* abort = reinterpret_cast<volatile int*>(tmem_holder + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < a.stages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int c = 0; c < 2; ++c) {
            mbar_init(&tfull[c], 1);
            mbar_init(&tempty[c], 4);
        }
        mbar_init(drain, 1);
        // (the 128B-swizzled stages need a 1024-byte aligned base)
        *abort = (smem_u32(smem_raw) & 1023u) != 0 ? 1 : 0;
        fence_mbar_init();
        prefetch_tmap(&tmap_x);
        prefetch_tmap(&tmap_x2);
        prefetch_tmap(&tmap_w);
    }
    if (warp == 1) tmem_alloc(tmem_holder, a.tmem_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    const int BM = 128 * a.mm;
    const int acc_cols = a.mm * a.npad;
    const int x_off = a.mm * GM_W_TILE;       // node rows after the weight rows in a stage
    // k-block range of split ks (the splits differ by at most one block)
    auto kb_lo = [&](int ks) { return (int)(((long)a.kblocks * ks) / a.KS); };

    if (warp == 0) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint64_t pol_w = policy_evict_first();
            const uint64_t pol_x = policy_evict_last();
            const uint32_t tx = (uint32_t)(BM * 128 + a.npad * 128);
            // node rows of k-block kb, from whichever input block holds it
            auto load_x = [&](uint8_t* dst, uint64_t* bar, int kb) {
                if (kb < a.kb_split)
                    tma_load_2d(dst, &tmap_x, bar, kb * 64, 0, pol_x);
                else
                    tma_load_2d(dst, &tmap_x2, bar, (kb - a.kb_split) * 64, 0, pol_x);
            };
            int s = 0;
            uint32_t ph = 0;
            int issued[8];
            for (int q = 0; q < 8; ++q) issued[q] = -1;
            // The first ring fill of W (a weight: no kernel of the stream
            // writes it) streams before the dependency wait; the node rows,
            // written upstream, are loaded after it.
            const int u0 = blockIdx.x;
            int pre = 0;
            if (u0 < a.units) {
                const int nt = u0 / a.KS, ks = u0 % a.KS;
                const int lo = kb_lo(ks), hi = kb_lo(ks + 1);
                pre = min(a.stages, hi - lo);
                for (int q = 0; q < pre; ++q) {
                    mbar_arrive_expect_tx(&full[q], tx);
                    tma_load_2d(stage_base + (size_t)q * a.stage_bytes, &tmap_w, &full[q], (lo + q) * 64, nt * BM,
                                pol_w);
                    issued[q] = 0;
                }
            }
            pdl_wait();
            pdl_trigger();
            if (u0 < a.units) {
                const int lo = kb_lo(u0 % a.KS);
                for (int q = 0; q < pre; ++q) load_x(stage_base + (size_t)q * a.stage_bytes + x_off, &full[q], lo + q);
            }
            s = pre % a.stages;
            ph = pre == a.stages ? 1u : 0u;
            for (int u = blockIdx.x; u < a.units; u += gridDim.x) {
                const int nt = u / a.KS, ks = u % a.KS;
                const int lo = kb_lo(ks), hi = kb_lo(ks + 1);
                for (int kb = lo + (u == u0 ? pre : 0); kb < hi; ++kb) {
                    if (!mbar_wait(&empty[s], ph ^ 1u, abort)) goto producer_done;
                    mbar_arrive_expect_tx(&full[s], tx);
                    uint8_t* st = stage_base + (size_t)s * a.stage_bytes;
                    tma_load_2d(st, &tmap_w, &full[s], kb * 64, nt * BM, pol_w);
                    load_x(st + x_off, &full[s], kb);
                    issued[s] = (int)ph;
                    if (++s == a.stages) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
            }
        producer_done:
            if (*abort) {
                for (int q = 0; q < a.stages; ++q)
                    if (issued[q] >= 0) mbar_wait_timeout_only(&full[q], (uint32_t)issued[q]);
            }
        }
    } else if (warp == 1) {
        // -------------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(128, a.npad);
            int s = 0;
            uint32_t ph = 0;
            int i = 0;
            for (int u = blockIdx.x; u < a.units; u += gridDim.x, ++i) {
                const int ks = u % a.KS;
                const int lo = kb_lo(ks), hi = kb_lo(ks + 1);
                const int acc = i & 1;
                if (!mbar_wait(&tempty[acc], ((uint32_t)(i >> 1) & 1u) ^ 1u, abort)) break;
                tc_fence_after();
                const uint32_t d_base = tmem + (uint32_t)(acc * acc_cols);
                bool ok = true;
                for (int kb = lo; kb < hi; ++kb) {
                    if (!mbar_wait(&full[s], ph, abort)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    uint8_t* st = stage_base + (size_t)s * a.stage_bytes;
                    const uint64_t bdesc = sdesc_kmajor_sw128(smem_u32(st + x_off));
                    for (int m = 0; m < a.mm; ++m) {
                        const uint64_t adesc = sdesc_kmajor_sw128(smem_u32(st + m * GM_W_TILE));
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            mma_bf16(d_base + (uint32_t)(m * a.npad), adesc + 2u * kk, bdesc + 2u * kk, idesc,
                                     (kb != lo || kk != 0) ? 1u : 0u);
                    }
                    mma_commit(&empty[s]);
                    if (++s == a.stages) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
                if (!ok) break;
                mma_commit(&tfull[acc]);
            }
            mma_commit(drain);
            mbar_wait_timeout_only(drain, 0);
        }
    } else {
        // ----------------------------------------------------------- epilogue
        // TMEM lane = weight row (output column n), TMEM column = node row r.
        const int sub = warp & 3;                 // TMEM lane quarter this warp may access
        pdl_wait();   // (before this role's global writes)
        if constexpr (CSK) {
            // The CTA's one unit: stage its fp32 sums as stage[node row][tile column]
            // over the (now idle) stage ring, for the cluster's reduction.
            int ok = 1;
            if (lane == 0) ok = mbar_wait(&tfull[0], 0, abort);
            ok = __shfl_sync(FULL, ok, 0);
            __syncwarp();
            tc_fence_after();
            float* stg = reinterpret_cast<float*>(smem_raw);
            if (ok) {
                for (int m = 0; m < a.mm; ++m) {
                    const int nl = m * 128 + sub * 32 + lane;
                    for (int c0 = 0; c0 < a.npad; c0 += 32) {
                        uint32_t v[32];
                        tmem_ld32(tmem + ((uint32_t)(sub * 32) << 16) + (uint32_t)(m * a.npad + c0), v);
                        tmem_wait_ld();
#pragma unroll
                        for (int j = 0; j < 32; ++j) stg[(size_t)(c0 + j) * BM + nl] = __uint_as_float(v[j]);
                    }
                }
            }
            tc_fence_before();
        } else {
        // Once a wait gives up, this CTA's remaining tiles get NaN partials,
        // so that the reduction turns the affected outputs into NaN.
        bool failed = false;
        int i = 0;
        for (int u = blockIdx.x; u < a.units; u += gridDim.x, ++i) {
            const int nt = u / a.KS, ks = u % a.KS;
            const int acc = i & 1;
            if (!failed) {
                int ok = 1;
                if (lane == 0) ok = mbar_wait(&tfull[acc], (uint32_t)(i >> 1) & 1u, abort);
                failed = __shfl_sync(FULL, ok, 0) == 0;
            }
            __syncwarp();
            tc_fence_after();
            for (int m = 0; m < a.mm; ++m) {
                const int n = nt * BM + m * 128 + sub * 32 + lane;
                float* dst = a.part + (size_t)ks * a.rows * a.N + n;
                for (int c0 = 0; c0 < a.npad; c0 += 32) {
                    uint32_t v[32];
                    if (!failed) {
                        tmem_ld32(tmem + ((uint32_t)(sub * 32) << 16) + (uint32_t)(acc * acc_cols + m * a.npad + c0),
                                  v);
                        tmem_wait_ld();
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j) v[j] = __float_as_uint(NAN);
                    }
                    if (n < a.N) {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (c0 + j < a.rows) dst[(size_t)(c0 + j) * a.N] = __uint_as_float(v[j]);
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0 && !failed) mbar_arrive(&tempty[acc]);
        }
        }
    }

    if constexpr (CSK) {
        // All CTAs of the cluster have staged their split's sums; CTA `rank`
        // reduces its share of the tile's columns (8-column chunks
        // [rank * BM/8 / KS, (rank + 1) * BM/8 / KS)) over the splits in rank
        // order (deterministic), applies the epilogue and writes bf16.  A
        // split that gave up makes the outputs NaN.
        pdl_wait();
        __syncthreads();
        cluster_sync_all();
        const uint32_t rank = cluster_rank();
        const int nt = blockIdx.x / a.KS;
        // this rank's 8-column chunks of the tile (the ranks split BM / 8 chunks
        // as evenly as they go; the planner forms clusters of 2 and 4 only,
        // which divide BM / 8, so an uneven split is not reached from the API)
        const int nch = BM / 8;
        const int c_lo = (int)rank * nch / a.KS, chunks = ((int)rank + 1) * nch / a.KS - c_lo;
        const uint32_t stg0 = smem_u32(smem_raw), ab0 = smem_u32((const void*)abort);
        bool bad = false;
        for (int p = 0; p < a.KS; ++p) bad |= ld_dsmem_s32(dsmem_addr(ab0, (uint32_t)p)) != 0;
        for (int it = threadIdx.x; it < a.rows * chunks; it += GM_THREADS) {
            const int r = it / chunks, nl = (c_lo + (it - r * chunks)) * 8;
            const int n = nt * BM + nl;
            if (n >= a.N) continue;
            float acc[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[e] = 0.f;
            if (a.bias) bf16x8_add(acc, a.bias + n);
            const uint32_t off = (uint32_t)(((size_t)r * BM + nl) * 4);
            for (int p = 0; p < a.KS; ++p) {
                const uint32_t q = dsmem_addr(stg0 + off, (uint32_t)p);
                const float4 v0 = ld_dsmem_f4(q), v1 = ld_dsmem_f4(q + 16);
                acc[0] += v0.x; acc[1] += v0.y; acc[2] += v0.z; acc[3] += v0.w;
                acc[4] += v1.x; acc[5] += v1.y; acc[6] += v1.z; acc[7] += v1.w;
            }
            if (a.epi == GV_LINEAR_SILU) {
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[e] = acc[e] / (1.0f + __expf(-acc[e]));
            } else if (a.epi == GV_LINEAR_ADD) {
                bf16x8_add(acc, a.residual + (size_t)r * a.n_out + n);
            }
            if (bad) {
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[e] = NAN;
            }
            uint32_t pk[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                __nv_bfloat162 h2 = __floats2bfloat162_rn(acc[2 * e], acc[2 * e + 1]);
                pk[e] = *reinterpret_cast<uint32_t*>(&h2);
            }
            const OutSplit& os = a.os;
            __nv_bfloat16* dst;
            if (os.n1 == 0 || n < os.n0)
                dst = os.out0 + (size_t)r * (os.n1 == 0 ? a.n_out : os.n0) + n;
            else if (n < os.n0 + os.n1)
                dst = os.out1 + (size_t)r * os.n1 + (n - os.n0);
            else
                dst = os.out2 + (size_t)r * (a.n_out - os.n0 - os.n1) + (n - os.n0 - os.n1);
            *reinterpret_cast<uint4*>(dst) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        }
        __syncwarp();
        cluster_sync_all();        // (no CTA leaves while a peer may still read its shared memory)
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, a.tmem_cols);
}

__global__ void __launch_bounds__(256)
gemm_reduce_kernel(const float* __restrict__ part, int KS, int rows, int N, int n_out, int epi,
                   const __nv_bfloat16* __restrict__ bias, const __nv_bfloat16* residual, OutSplit os) {
    pdl_trigger();   // (early: see the split-K reduce note in gv_internal.cuh)
    pdl_wait();
    const int per_row = n_out / 8;
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= rows * per_row) return;
    const int r = idx / per_row, c = (idx - r * per_row) * 8;
    float acc[8], up[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] = up[e] = 0.f;
    if (bias) {
        bf16x8_add(acc, bias + c);
        if (epi == GV_LINEAR_SWIGLU) bf16x8_add(up, bias + n_out + c);
    }
#pragma unroll 4
    for (int ks = 0; ks < KS; ++ks) {
        const float* p = part + ((size_t)ks * rows + r) * N;
        const float4 a0 = *reinterpret_cast<const float4*>(p + c);
        const float4 a1 = *reinterpret_cast<const float4*>(p + c + 4);
        acc[0] += a0.x; acc[1] += a0.y; acc[2] += a0.z; acc[3] += a0.w;
        acc[4] += a1.x; acc[5] += a1.y; acc[6] += a1.z; acc[7] += a1.w;
        if (epi == GV_LINEAR_SWIGLU) {
            const float4 b0 = *reinterpret_cast<const float4*>(p + n_out + c);
            const float4 b1 = *reinterpret_cast<const float4*>(p + n_out + c + 4);
            up[0] += b0.x; up[1] += b0.y; up[2] += b0.z; up[3] += b0.w;
            up[4] += b1.x; up[5] += b1.y; up[6] += b1.z; up[7] += b1.w;
        }
    }
    float o[8];
    if (epi == GV_LINEAR_SWIGLU) {
#pragma unroll
        for (int e = 0; e < 8; ++e) o[e] = acc[e] / (1.0f + __expf(-acc[e])) * up[e];
    } else if (epi == GV_LINEAR_SILU) {
#pragma unroll
        for (int e = 0; e < 8; ++e) o[e] = acc[e] / (1.0f + __expf(-acc[e]));
    } else if (epi == GV_LINEAR_ADD) {
#pragma unroll
        for (int e = 0; e < 8; ++e) o[e] = acc[e];
        bf16x8_add(o, residual + (size_t)r * n_out + c);
    } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) o[e] = acc[e];
    }
    uint32_t pk[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        __nv_bfloat162 h2 = __floats2bfloat162_rn(o[2 * e], o[2 * e + 1]);
        pk[e] = *reinterpret_cast<uint32_t*>(&h2);
    }
    __nv_bfloat16* dst;
    if (os.n1 == 0 || c < os.n0)
        dst = os.out0 + (size_t)r * (os.n1 == 0 ? n_out : os.n0) + c;
    else if (c < os.n0 + os.n1)
        dst = os.out1 + (size_t)r * os.n1 + (c - os.n0);
    else
        dst = os.out2 + (size_t)r * (n_out - os.n0 - os.n1) + (c - os.n0 - os.n1);
    *reinterpret_cast<uint4*>(dst) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
}

// The residual-add epilogue fused with the RMSNorm that follows it in the
// layer: one CTA per row adds the K splits and the residual, writes the bf16
// row h, and from the stored (rounded) values writes
// norm_out = h / sqrt(mean(h^2) + eps) * w.  n_out % 8 == 0, n_out <= 8192.
// Each thread owns RN_MAXC 16-byte chunks of the row; the split loop runs
// over all of them at once, so that a thread has up to 4 * RN_MAXC * 2 loads
// of partial sums in flight (the partials sit in L2: the loop is latency-,
// not bandwidth-bound).
constexpr int RN_THREADS = 512;
constexpr int RN_MAXC = 2;                         // n_out <= RN_THREADS * RN_MAXC * 8

__global__ void __launch_bounds__(RN_THREADS)
gemm_reduce_norm_kernel(const float* __restrict__ part, int KS, int rows, int n_out,
                        const __nv_bfloat16* residual, __nv_bfloat16* out, const __nv_bfloat16* __restrict__ w,
                        float eps, __nv_bfloat16* __restrict__ norm_out) {
    __shared__ float red[RN_THREADS / 32];
    pdl_trigger();   // (early: see the split-K reduce note in gv_internal.cuh)
    pdl_wait();
    const int r = blockIdx.x, tid = threadIdx.x;
    float acc[RN_MAXC][8];
#pragma unroll
    for (int q = 0; q < RN_MAXC; ++q) {
        const int c = (tid + q * RN_THREADS) * 8;
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[q][e] = 0.f;
        if (c < n_out) bf16x8_add(acc[q], residual + (size_t)r * n_out + c);
    }
#pragma unroll 4
    for (int ks = 0; ks < KS; ++ks) {
        const float* prow = part + ((size_t)ks * rows + r) * n_out;
#pragma unroll
        for (int q = 0; q < RN_MAXC; ++q) {
            const int c = (tid + q * RN_THREADS) * 8;
            if (c < n_out) {
                const float4 a0 = *reinterpret_cast<const float4*>(prow + c);
                const float4 a1 = *reinterpret_cast<const float4*>(prow + c + 4);
                acc[q][0] += a0.x; acc[q][1] += a0.y; acc[q][2] += a0.z; acc[q][3] += a0.w;
                acc[q][4] += a1.x; acc[q][5] += a1.y; acc[q][6] += a1.z; acc[q][7] += a1.w;
            }
        }
    }
    float ss = 0.f;
#pragma unroll
    for (int q = 0; q < RN_MAXC; ++q) {
        const int c = (tid + q * RN_THREADS) * 8;
        if (c >= n_out) break;
        uint32_t pk[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            __nv_bfloat162 h2 = __floats2bfloat162_rn(acc[q][2 * e], acc[q][2 * e + 1]);
            pk[e] = *reinterpret_cast<uint32_t*>(&h2);
            acc[q][2 * e] = __uint_as_float(pk[e] << 16);          // the stored (rounded) h
            acc[q][2 * e + 1] = __uint_as_float(pk[e] & 0xffff0000u);
            ss += acc[q][2 * e] * acc[q][2 * e] + acc[q][2 * e + 1] * acc[q][2 * e + 1];
        }
        *reinterpret_cast<uint4*>(out + (size_t)r * n_out + c) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
    }
    ss = warp_sum(ss);
    if ((tid & 31) == 0) red[tid >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int k = 0; k < RN_THREADS / 32; ++k) tot += red[k];
    const float inv = rsqrtf(tot / (float)n_out + eps);
#pragma unroll
    for (int q = 0; q < RN_MAXC; ++q) {
        const int c = (tid + q * RN_THREADS) * 8;
        if (c >= n_out) break;
        const uint4 g = *reinterpret_cast<const uint4*>(w + c);
        const uint32_t gw[4] = {g.x, g.y, g.z, g.w};
        uint32_t pk[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            __nv_bfloat162 h2 = __floats2bfloat162_rn(acc[q][2 * e] * inv * __uint_as_float(gw[e] << 16),
                                                      acc[q][2 * e + 1] * inv * __uint_as_float(gw[e] & 0xffff0000u));
            pk[e] = *reinterpret_cast<uint32_t*>(&h2);
        }
        *reinterpret_cast<uint4*>(norm_out + (size_t)r * n_out + c) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
    }
}

// RMSNorm of one row per CTA: out = x / sqrt(mean(x^2) + eps) * w, fp32 math,
// bf16 in and out (16-byte vectors; H % 8 == 0).
__global__ void __launch_bounds__(256)
rmsnorm_kernel(const __nv_bfloat16* __restrict__ x, const __nv_bfloat16* __restrict__ w, int H, float eps,
               __nv_bfloat16* __restrict__ out) {
    __shared__ float red[8];
    pdl_wait();
    pdl_trigger();
    const int r = blockIdx.x, tid = threadIdx.x;
    const uint4* xr = reinterpret_cast<const uint4*>(x + (size_t)r * H);
    float ss = 0.f;
    for (int i = tid; i < H / 8; i += blockDim.x) {
        const uint4 v = xr[i];
        const uint32_t q[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float lo = __uint_as_float(q[e] << 16), hi = __uint_as_float(q[e] & 0xffff0000u);
            ss += lo * lo + hi * hi;
        }
    }
    ss = warp_sum(ss);
    if ((tid & 31) == 0) red[tid >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) tot += red[k];
    const float inv = rsqrtf(tot / (float)H + eps);
    const uint4* wr = reinterpret_cast<const uint4*>(w);
    uint4* orow = reinterpret_cast<uint4*>(out + (size_t)r * H);
    for (int i = tid; i < H / 8; i += blockDim.x) {
        const uint4 v = xr[i], g = wr[i];
        const uint32_t q[4] = {v.x, v.y, v.z, v.w}, gw[4] = {g.x, g.y, g.z, g.w};
        uint32_t pk[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float lo = __uint_as_float(q[e] << 16) * inv * __uint_as_float(gw[e] << 16);
            const float hi = __uint_as_float(q[e] & 0xffff0000u) * inv * __uint_as_float(gw[e] & 0xffff0000u);
            __nv_bfloat162 h2 = __floats2bfloat162_rn(lo, hi);
            pk[e] = *reinterpret_cast<uint32_t*>(&h2);
        }
        orow[i] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
    }
}

// ----------------------------------------------------------------- host side
// Split-K through global memory: (mm, KS) minimising ceil(units / SMs) * per-unit
// cost, a unit's cost counted in rows streamed per k-block (BM weight rows +
// npad node rows) plus an epilogue share; larger tiles on ties.  Cluster
// split-K (the KS CTAs of a tile in one cluster, KS in {2, 4}, one wave) costs
// ceil(kblocks / KS) * (BM + npad) + BM, scaled by SMs / CTAs, and saves the
// partial sums' round trip through L2 and the reduce launch (counted as
// GM_REDUCE_COST).  With 60 node rows this picks the cluster form for the O
// projection (4096 x 4096) and the drafter's fusion projections (4096 x 8192,
// 4096 x 11008), where it measured 0.6-1.1 us faster, and the global form for
// the Q/K/V (6144 x 4096) and down (4096 x 14336) projections, where the
// cluster form measured 0.4-0.8 us slower.  (Other cluster sizes -- the
// kernel splits a tile's columns unevenly when KS does not divide BM / 8 --
// measured no better: Q/K/V in clusters of 5 took 17.7 us against 17.1, the
// 11008 x 8192 fusion projection in clusters of 3 took 39.0 us against the
// global form's ~35.)
struct GemmPlan {
    int mm, KS, n_tiles, kblocks, units, grid, npad;
    bool csk;
};

int launch_rmsnorm(const void* x, const void* w, int rows, int H, float eps, void* out, cudaStream_t st);

constexpr int GM_SMEM_BUDGET = 220 * 1024;
constexpr long GM_REDUCE_COST = 3500;

static int gemm_stage_bytes(int mm, int npad) { return mm * GM_W_TILE + npad * 128; }
static int gemm_stages(int stage_bytes) {
    const int n = (GM_SMEM_BUDGET - 2048) / stage_bytes;
    return n > 8 ? 8 : n;
}
static size_t gemm_smem(int stages, int stage_bytes) { return (size_t)stages * stage_bytes + 8 * (2 * stages + 5) + 16; }

// Clusters of c CTAs of the cluster split-K kernel resident at once (0 if
// the device cannot say), per (c, shared memory size).
static int gemm_max_clusters(int c, size_t smem) {
    static std::map<std::pair<int, size_t>, int> cache;
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    const auto key = std::make_pair(c, smem);
    auto it = cache.find(key);
    if (it != cache.end()) return it->second;
    int n = 0;
    if (cudaFuncSetAttribute(gemm_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) ==
        cudaSuccess) {
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = (unsigned)c;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3((unsigned)(c * 16));
        cfg.blockDim = dim3(GM_THREADS);
        cfg.dynamicSmemBytes = smem;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        if (cudaOccupancyMaxActiveClusters(&n, gemm_tc_kernel<true>, &cfg) != cudaSuccess) n = 0;
    }
    cudaGetLastError();
    cache[key] = n;
    return n;
}

static GemmPlan gemm_plan(int rows, int N, int K, bool allow_csk) {
    const int npad = (rows + 31) / 32 * 32;
    const int sms = sm_count();
    GemmPlan best{};
    long best_cost = -1;
    const int kblocks = (K + 63) / 64;
    for (int mm = 1; mm <= 2 && 2 * mm * npad <= 512; ++mm) {
        const int bm = 128 * mm;
        const int tiles = (N + bm - 1) / bm;
        for (int ks = 1; ks <= kblocks && ks <= 32; ++ks) {
            const long units = (long)tiles * ks;
            const long waves = (units + sms - 1) / sms;
            const long kb_per = (kblocks + ks - 1) / ks;
            const long cost = waves * (kb_per * (bm + npad) + 2L * bm) + GM_REDUCE_COST;
            if (best_cost < 0 || cost < best_cost || (cost == best_cost && mm > best.mm)) {
                best_cost = cost;
                best = GemmPlan{mm, ks, tiles, kblocks, (int)units, 0, npad, false};
            }
        }
    }
    best.grid = best.units < sms ? best.units : sms;
    if (!allow_csk) return best;
    for (int mm = 1; mm <= 2 && 2 * mm * npad <= 512; ++mm) {
        const int bm = 128 * mm;
        const int tiles = (N + bm - 1) / bm;
        const int sb = gemm_stage_bytes(mm, npad), st = gemm_stages(sb);
        if ((size_t)npad * bm * 4 > (size_t)st * sb) continue;        // the staged sums must fit the ring
        for (int c = 2; c <= 4; c += 2) {
            if (c > kblocks || tiles > gemm_max_clusters(c, gemm_smem(st, sb))) continue;
            // (scaled by the SMs left idle: one SM streams only so fast, so fewer
            // CTAs take proportionally longer)
            const long ctas = (long)tiles * c;
            const long cost = ((long)((kblocks + c - 1) / c) * (bm + npad) + bm) * sms / (ctas < sms ? ctas : sms);
            if (cost < best_cost) {
                best_cost = cost;
                best = GemmPlan{mm, c, tiles, kblocks, tiles * c, tiles * c, npad, true};
            }
        }
    }
    return best;
}

size_t linear_workspace_bytes(int rows, int K, int N) {
    const GemmPlan p = gemm_plan(rows, N, K, false);     // (an upper bound of what any plan needs)
    return (size_t)p.KS * rows * N * sizeof(float);
}

static GemmArgs gemm_args(const LinearOp& op, const GemmPlan& p, int N) {
    GemmArgs a{};
    a.rows = op.rows;
    a.npad = p.npad;
    a.N = N;
    a.K = op.K;
    a.mm = p.mm;
    a.n_tiles = p.n_tiles;
    a.KS = p.KS;
    a.kblocks = p.kblocks;
    a.units = p.units;
    a.stage_bytes = gemm_stage_bytes(a.mm, a.npad);
    a.stages = gemm_stages(a.stage_bytes);
    const int cols = 2 * a.mm * a.npad;
    a.tmem_cols = cols <= 32 ? 32 : cols <= 64 ? 64 : cols <= 128 ? 128 : cols <= 256 ? 256 : 512;
    a.part = static_cast<float*>(op.ws);
    a.kb_split = op.x2 ? op.k_split / 64 : a.kblocks;
    a.n_out = op.n_out;
    a.epi = op.epi;
    a.bias = static_cast<const __nv_bfloat16*>(op.bias);
    a.residual = static_cast<const __nv_bfloat16*>(op.residual);
    a.os = OutSplit{static_cast<__nv_bfloat16*>(op.out), static_cast<__nv_bfloat16*>(op.out1),
                    static_cast<__nv_bfloat16*>(op.out2), op.n0, op.n1};
    return a;
}

static int gemm_maps(const LinearOp& op, const GemmArgs& a, CUtensorMap* mx, CUtensorMap* mx2, CUtensorMap* mw) {
    // one input block: x2's map is never read (kb_split = kblocks)
    const int k1 = op.x2 ? op.k_split : op.K;
    int rc = make_map_2d(mx, op.x, (uint64_t)op.rows, (uint64_t)k1, (uint32_t)a.npad, (uint64_t)k1 * 2);
    if (rc != GV_OK) return rc;
    if (op.x2) {
        const int k2 = op.K - op.k_split;
        rc = make_map_2d(mx2, op.x2, (uint64_t)op.rows, (uint64_t)k2, (uint32_t)a.npad, (uint64_t)k2 * 2);
        if (rc != GV_OK) return rc;
    } else {
        *mx2 = *mx;
    }
    return make_map_2d(mw, op.W, (uint64_t)a.N, (uint64_t)op.K, (uint32_t)(128 * a.mm), (uint64_t)op.K * 2);
}

int launch_gemm_partials(const LinearOp& op, cudaStream_t st, int* ks) {
    const int N = op.epi == GV_LINEAR_SWIGLU ? 2 * op.n_out : op.n_out;
    const GemmPlan p = gemm_plan(op.rows, N, op.K, false);
    GemmArgs a = gemm_args(op, p, N);
    CUtensorMap mx, mx2, mw;
    int rc = gemm_maps(op, a, &mx, &mx2, &mw);
    if (rc != GV_OK) return rc;
    const size_t smem = gemm_smem(a.stages, a.stage_bytes);
    cudaFuncSetAttribute(gemm_tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    launch_pdl(gemm_tc_kernel<false>, dim3(p.grid), dim3(GM_THREADS), smem, st, mx, mx2, mw, a);
    *ks = a.KS;
    return check_launch("gemm_tc_kernel");
}

// The cluster split-K form: one launch writes the epilogue's bf16 output.
static int launch_gemm_csk(const LinearOp& op, const GemmPlan& p, cudaStream_t st) {
    GemmArgs a = gemm_args(op, p, op.n_out);
    CUtensorMap mx, mx2, mw;
    int rc = gemm_maps(op, a, &mx, &mx2, &mw);
    if (rc != GV_OK) return rc;
    const size_t smem = gemm_smem(a.stages, a.stage_bytes);
    cudaFuncSetAttribute(gemm_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = (unsigned)a.KS;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3((unsigned)p.grid);
    cfg.blockDim = dim3(GM_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    cudaLaunchKernelEx(&cfg, gemm_tc_kernel<true>, mx, mx2, mw, a);
    return check_launch("gemm_tc_kernel (cluster split-K)");
}

int launch_linear(const LinearOp& op, cudaStream_t st) {
    const int N = op.epi == GV_LINEAR_SWIGLU ? 2 * op.n_out : op.n_out;
    if (op.epi != GV_LINEAR_SWIGLU) {
        const GemmPlan p = gemm_plan(op.rows, N, op.K, true);
        if (p.csk) {
            int rc = launch_gemm_csk(op, p, st);
            if (rc != GV_OK || !op.norm_out) return rc;
            return launch_rmsnorm(op.out, op.norm_w, op.rows, op.n_out, op.eps, op.norm_out, st);
        }
    }
    int KS = 0;
    int rc = launch_gemm_partials(op, st, &KS);
    if (rc != GV_OK) return rc;
    const float* part = static_cast<const float*>(op.ws);
    if (op.norm_out) {
        launch_pdl(gemm_reduce_norm_kernel, dim3(op.rows), dim3(RN_THREADS), 0, st, part, KS, op.rows, op.n_out,
                   static_cast<const __nv_bfloat16*>(op.residual), static_cast<__nv_bfloat16*>(op.out),
                   static_cast<const __nv_bfloat16*>(op.norm_w), op.eps, static_cast<__nv_bfloat16*>(op.norm_out));
        return check_launch("gemm_reduce_norm_kernel");
    }
    const int items = op.rows * (op.n_out / 8);
    OutSplit os{static_cast<__nv_bfloat16*>(op.out), static_cast<__nv_bfloat16*>(op.out1),
                static_cast<__nv_bfloat16*>(op.out2), op.n0, op.n1};
    launch_pdl(gemm_reduce_kernel, dim3((items + 255) / 256), dim3(256), 0, st, part, KS, op.rows, N, op.n_out,
               op.epi, static_cast<const __nv_bfloat16*>(op.bias), static_cast<const __nv_bfloat16*>(op.residual),
               os);
    return check_launch("gemm_reduce_kernel");
}

int launch_rmsnorm(const void* x, const void* w, int rows, int H, float eps, void* out, cudaStream_t st) {
    launch_pdl(rmsnorm_kernel, dim3(rows), dim3(256), 0, st, static_cast<const __nv_bfloat16*>(x),
               static_cast<const __nv_bfloat16*>(w), H, eps, static_cast<__nv_bfloat16*>(out));
    return check_launch("rmsnorm_kernel");
}

}  // namespace gv
