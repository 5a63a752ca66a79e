// gv_lmhead_select, bf16 tensor-core path for sm_103a.
//
// GRIFFIN Section 3 / Eq. 1: the LM head maps each draft node's final hidden
// state to vocabulary scores; greedy verification (Section 5, T = 0) needs
// only each node's argmax, so the scores are reduced on chip and never
// written (the paper's closing remark on fusing kernels to cut memory
// traffic).  The weight W[V][H] is read from HBM exactly once.
//
// One persistent CTA per SM takes a contiguous range of the vocabulary: the
// V rows, in groups of 16, are cut into as many equal ranges as CTAs (they
// differ by at most one group), and a CTA's range into `tpc` tiles of k or
// k + 1 groups.  Per tile:  S[r][v] = sum_k h[r][k] W[v][k]  with the hidden
// rows on the MMA M side (128 rows per M tile, rows beyond `rows` are
// zero-filled by TMA) and the tile's vocabulary rows on the N side (one
// tensor map per tile height), both operands K-major with the 128-byte
// swizzle, fp32 accumulators in tensor memory, double-buffered so the MMA of
// tile i+1 overlaps the epilogue of tile i.
//
// Warp roles (192 threads):
//   warp 0     one lane issues TMA loads of h and W k-blocks into a ring of
//              shared-memory stages (W with an evict-first L2 hint, h with
//              evict-last: h is re-read for every tile, W never);
//   warp 1     allocates TMEM; one lane issues tcgen05.mma and commits each
//              stage back to the producer and each finished tile to the
//              epilogue;
//   warps 2-5  one thread per M-tile row (TMEM lane): read the tile's scores
//              32 columns at a time and fold them into a running per-row
//              argmax / top-K / (max, sum exp) state; logits mode also stores
//              the scores.
// Each CTA finally writes its per-row partial result to the workspace, and
// lmhead_merge_kernel combines the CTAs' partials.  Every wait is bounded.
#include "gv_internal.cuh"
#include "sm103.cuh"

namespace gv {
using namespace sm103;

constexpr int LM_THREADS = 192;
constexpr int LM_A_TILE_BYTES = 128 * 128;   // 128 rows x 64 bf16
constexpr int LM_PRE_STAGES = 8;             // W stages issued before the dependency wait (the ring)

struct LmTcArgs {
    int rows;          // rows of this launch (<= 256)
    int row0;          // first global row of this launch (partials are indexed globally)
    int V, mt, kblocks, stages, stage_bytes;
    int groups;        // 16-row vocabulary groups, ceil(V / 16)
    int tpc;           // tiles per CTA
    int bn_small;      // rows of the smaller tile height (tmap_ws), 0 if there is none
    int bn_max;        // rows of the larger tile height (tmap_wb): TMEM columns per M tile
    int a_bytes;       // hidden-row bytes per stage (see launch_lmhead_tc)
    uint32_t tmem_cols;
    int mode, K;
    float* logits;     // [rows_total][V] (mode LOGITS)
    SelectPartials part;
    int* err;          // [grid] per-CTA status: 0, or GV_ERR_TIMEOUT after a bounded wait gave up
};

// Tile i of this CTA: vocabulary rows [v0, v0 + n); n = 0 means no tile.
struct LmTile {
    int v0, n;
};
__device__ __forceinline__ LmTile lm_tile(const LmTcArgs& a, int i) {
    const int C = gridDim.x, c = blockIdx.x;
    const int gc0 = (int)((long long)c * a.groups / C);
    const int gcn = (int)((long long)(c + 1) * a.groups / C) - gc0;
    const int g0 = gc0 + (int)((long long)gcn * i / a.tpc);
    const int g1 = gc0 + (int)((long long)gcn * (i + 1) / a.tpc);
    return {g0 * 16, (g1 - g0) * 16};
}

template <int KM>
__global__ void __launch_bounds__(LM_THREADS, 1)
lmhead_tc_kernel(const __grid_constant__ CUtensorMap tmap_h, const __grid_constant__ CUtensorMap tmap_ws,
                 const __grid_constant__ CUtensorMap tmap_wb, LmTcArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~static_cast<uintptr_t>(1023));
    uint8_t* stage_base = smem;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)a.stages * a.stage_bytes);
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
        *abort = 0;
        fence_mbar_init();
        prefetch_tmap(&tmap_h);
        prefetch_tmap(&tmap_ws);
        prefetch_tmap(&tmap_wb);
    }
    if (warp == 1) tmem_alloc(tmem_holder, a.tmem_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    const int acc_cols = a.mt * a.bn_max;
    // (the map of a tile's height)
    auto wmap = [&](int n) { return n == a.bn_small ? &tmap_ws : &tmap_wb; };

    if (warp == 0) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint64_t pol_w = policy_evict_first();
            const uint64_t pol_h = policy_evict_last();
            int s = 0;
            uint32_t ph = 0;
            int issued[8];   // parity of the last load issued into each stage, or -1
            for (int q = 0; q < 8; ++q) issued[q] = -1;
            // The first W stages (a weight: no kernel of the stream writes it)
            // stream before the dependency wait; the hidden rows, written
            // upstream, are loaded after it.  The whole ring: CTAs that start
            // during the preceding kernel's tail fill it while HBM is idle
            // (2 stages measured 2 us slower on the whole verify step).
            int i0 = 0;
            LmTile t0 = lm_tile(a, 0);
            while (t0.n == 0 && ++i0 < a.tpc) t0 = lm_tile(a, i0);
            const int pre = t0.n > 0 ? min(LM_PRE_STAGES, a.stages < a.kblocks ? a.stages : a.kblocks) : 0;
            for (int q = 0; q < pre; ++q) {
                mbar_arrive_expect_tx(&full[q], (uint32_t)(a.a_bytes + t0.n * 128));
                tma_load_2d(stage_base + (size_t)q * a.stage_bytes + a.a_bytes, wmap(t0.n), &full[q], q * 64,
                            t0.v0, pol_w);
                issued[q] = 0;
            }
            pdl_wait();
            pdl_trigger();
            for (int q = 0; q < pre; ++q)
                for (int m = 0; m < a.mt; ++m)
                    tma_load_2d(stage_base + (size_t)q * a.stage_bytes + m * LM_A_TILE_BYTES, &tmap_h,
                                &full[q], q * 64, m * 128, pol_h);
            s = pre % a.stages;
            ph = pre == a.stages ? 1u : 0u;
            for (int ti = i0; ti < a.tpc; ++ti) {
                const LmTile tl = lm_tile(a, ti);
                if (tl.n == 0) continue;
                const uint32_t tx = (uint32_t)(a.a_bytes + tl.n * 128);
                for (int kb = ti == i0 ? pre : 0; kb < a.kblocks; ++kb) {
                    if (!mbar_wait(&empty[s], ph ^ 1u, abort)) goto producer_done;
                    mbar_arrive_expect_tx(&full[s], tx);
                    uint8_t* st = stage_base + (size_t)s * a.stage_bytes;
                    for (int m = 0; m < a.mt; ++m)
                        tma_load_2d(st + m * LM_A_TILE_BYTES, &tmap_h, &full[s], kb * 64, m * 128, pol_h);
                    tma_load_2d(st + a.a_bytes, wmap(tl.n), &full[s], kb * 64, tl.v0, pol_w);
                    issued[s] = (int)ph;
                    if (++s == a.stages) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
            }
        producer_done:
            // On abort, let the copies this thread issued land before the CTA
            // exits (each wait bounded on its own).
            if (*abort) {
                for (int q = 0; q < a.stages; ++q)
                    if (issued[q] >= 0) mbar_wait_timeout_only(&full[q], (uint32_t)issued[q]);
            }
        }
    } else if (warp == 1) {
        // -------------------------------------------------------- MMA issuer
        if (lane == 0) {
            int s = 0;
            uint32_t ph = 0;
            int i = 0;      // tiles with rows so far
            for (int ti = 0; ti < a.tpc; ++ti) {
                const LmTile tl = lm_tile(a, ti);
                if (tl.n == 0) continue;
                const uint32_t idesc = idesc_bf16(128, tl.n);
                const int acc = i & 1;
                if (!mbar_wait(&tempty[acc], ((uint32_t)(i >> 1) & 1u) ^ 1u, abort)) break;
                tc_fence_after();
                const uint32_t d_base = tmem + (uint32_t)(acc * acc_cols);
                bool ok = true;
                for (int kb = 0; kb < a.kblocks; ++kb) {
                    if (!mbar_wait(&full[s], ph, abort)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    uint8_t* st = stage_base + (size_t)s * a.stage_bytes;
                    const uint64_t bdesc = sdesc_kmajor_sw128(smem_u32(st + a.a_bytes));
                    for (int m = 0; m < a.mt; ++m) {
                        const uint64_t adesc = sdesc_kmajor_sw128(smem_u32(st + m * LM_A_TILE_BYTES));
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            mma_bf16(d_base + (uint32_t)(m * a.bn_max), adesc + 2u * kk, bdesc + 2u * kk,
                                     idesc, (kb | kk) != 0);
                    }
                    mma_commit(&empty[s]);
                    if (++s == a.stages) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
                if (!ok) break;
                mma_commit(&tfull[acc]);
                ++i;
            }
            // Every MMA this thread issued has completed once `drain` flips.
            mma_commit(drain);
            mbar_wait_timeout_only(drain, 0);
        }
    } else {
        // ----------------------------------------------------------- epilogue
        const int sub = warp & 3;                 // TMEM lane quarter this warp may access
        const int row_in_tile = sub * 32 + lane;
        pdl_wait();   // (before this role's global writes: logits, partials)
        float lv[2][KM];
        int li[2][KM];
        float rm[2], rs[2];
#pragma unroll
        for (int m = 0; m < 2; ++m) {
            rm[m] = -INFINITY;
            rs[m] = 0.f;
#pragma unroll
            for (int q = 0; q < KM; ++q) {
                lv[m][q] = -INFINITY;
                li[m][q] = INT32_MAX;
            }
        }
        int i = 0;      // tiles with rows so far
        for (int ti = 0; ti < a.tpc; ++ti) {
            const LmTile tl = lm_tile(a, ti);
            if (tl.n == 0) continue;
            const int acc = i & 1;
            int ok = 1;
            if (lane == 0) ok = mbar_wait(&tfull[acc], (uint32_t)(i >> 1) & 1u, abort);
            ok = __shfl_sync(FULL, ok, 0);
            if (!ok) break;
            __syncwarp();
            tc_fence_after();
            const int v_tile = tl.v0;
            const int vlim = min(a.V, tl.v0 + tl.n);   // ids at or past it are not this tile's
#pragma unroll
            for (int m = 0; m < 2; ++m) {
                if (m >= a.mt) break;
                const int r = a.row0 + m * 128 + row_in_tile;
                const bool row_ok = m * 128 + row_in_tile < a.rows;
                for (int c0 = 0; c0 < tl.n; c0 += 32) {
                    uint32_t v[32];
                    const uint32_t taddr = tmem + ((uint32_t)(sub * 32) << 16) +
                                           (uint32_t)(acc * acc_cols + m * a.bn_max + c0);
                    if (c0 + 32 <= tl.n) {
                        tmem_ld32(taddr, v);
                    } else {
                        // a 16-column tail (tile heights are multiples of 16)
                        uint32_t v16[16];
                        tmem_ld16(taddr, v16);
#pragma unroll
                        for (int j = 0; j < 16; ++j) {
                            v[j] = v16[j];
                            v[16 + j] = 0u;
                        }
                    }
                    tmem_wait_ld();
                    const int id0 = v_tile + c0;
                    if (a.mode == GV_SELECT_LOGITS) {
                        float cmax = -INFINITY;
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (id0 + j < vlim) cmax = fmaxf(cmax, __uint_as_float(v[j]));
                        const float mnew = fmaxf(rm[m], cmax);
                        float sum = 0.f;
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (id0 + j < vlim) sum += __expf(__uint_as_float(v[j]) - mnew);
                        rs[m] = rs[m] * __expf(rm[m] - mnew) + sum;
                        rm[m] = mnew;
                        if (row_ok) {
                            float* dst = a.logits + (size_t)r * a.V + id0;
                            if (id0 + 32 <= vlim && (a.V & 3) == 0) {
#pragma unroll
                                for (int j = 0; j < 32; j += 4)
                                    *reinterpret_cast<float4*>(dst + j) = make_float4(
                                        __uint_as_float(v[j]), __uint_as_float(v[j + 1]),
                                        __uint_as_float(v[j + 2]), __uint_as_float(v[j + 3]));
                            } else {
                                for (int j = 0; j < 32 && id0 + j < vlim; ++j) dst[j] = __uint_as_float(v[j]);
                            }
                        }
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j) {
                            float cv = __uint_as_float(v[j]);
                            int ci = id0 + j;
                            // ids only grow, so a strict '>' keeps the lower id on ties
                            if (ci < vlim && cv > lv[m][KM - 1]) {
#pragma unroll
                                for (int q = 0; q < KM; ++q) {
                                    if (cv > lv[m][q]) {
                                        const float tv = lv[m][q];
                                        const int ti = li[m][q];
                                        lv[m][q] = cv;
                                        li[m][q] = ci;
                                        cv = tv;
                                        ci = ti;
                                    }
                                }
                            }
                        }
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[acc]);
            ++i;
        }
        // Per-CTA partial of every row this thread owns.
        const int slot = blockIdx.x;
#pragma unroll
        for (int m = 0; m < 2; ++m) {
            if (m >= a.mt) break;
            if (m * 128 + row_in_tile >= a.rows) continue;
            const int r = a.row0 + m * 128 + row_in_tile;
            const size_t pr = (size_t)slot * a.part.rows + r;
            if (a.mode == GV_SELECT_LOGITS) {
                a.part.m[pr] = rm[m];
                a.part.s[pr] = rm[m] == -INFINITY ? 0.f : rs[m];
            } else {
#pragma unroll
                for (int q = 0; q < KM; ++q) {
                    if (q < a.K) {
                        a.part.val[pr * a.K + q] = lv[m][q];
                        a.part.id[pr * a.K + q] = li[m][q];
                    }
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, a.tmem_cols);
    // Every CTA rewrites its status word each call (the first row chunk
    // clears it, any chunk may raise it), so no memset precedes the launch.
    if (threadIdx.x == 0) {
        if (*abort)
            a.err[blockIdx.x] = GV_ERR_TIMEOUT;
        else if (a.row0 == 0)
            a.err[blockIdx.x] = 0;
    }
}

// ----------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn tensor_map_encoder() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

// 2-D bf16 tensor map over a row-major [rows][cols] matrix, box [box_rows][64]
// with the 128-byte swizzle.
int make_map_2d(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows,
                uint64_t row_stride_bytes) {
    EncodeTiledFn enc = tensor_map_encoder();
    if (!enc) {
        set_error("cuTensorMapEncodeTiled unavailable");
        return GV_ERR_CUDA;
    }
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {row_stride_bytes};
    cuuint32_t box[2] = {64, box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                     box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        set_error("cuTensorMapEncodeTiled failed (%d)", (int)r);
        return GV_ERR_CUDA;
    }
    return GV_OK;
}

// Number of CTAs (= partial slots) the tensor-core LM head launches with.
int lmhead_tc_grid(int slots_capacity) {
    const int c = sm_count();
    return c < slots_capacity ? c : slots_capacity;
}

// Launches the kernel once per chunk of <= 256 rows; every launch uses the
// same grid, and a CTA with no vocabulary tile writes neutral partials, so
// the merge can read `grid` slots for every row.
int launch_lmhead_tc(const void* h, const void* W, int rows, int H, int V, int mode, int K,
                     float* logits, SelectPartials part, int* err, cudaStream_t st) {
    const int grid = part.slots;
    constexpr int SMEM_BUDGET = 220 * 1024;
    for (int row0 = 0; row0 < rows; row0 += 256) {
        const int r = rows - row0 < 256 ? rows - row0 : 256;
        LmTcArgs a{};
        a.rows = r;
        a.row0 = row0;
        a.V = V;
        a.mt = (r + 127) / 128;
        // Balanced vocabulary ranges: ceil(V / 16) groups of 16 rows cut into
        // `grid` ranges, each into tpc tiles of at most 16 / mt groups (TMEM:
        // two accumulators of mt x tile columns in 512); the tiles then have
        // kmin or kmin + 1 groups.
        a.groups = (V + 15) / 16;
        const int gmax_tile = 16 / a.mt;
        const int gcmax = (a.groups + grid - 1) / grid;
        a.tpc = std::max(1, (gcmax + gmax_tile - 1) / gmax_tile);
        const int kmin = (a.groups / grid) / a.tpc, kmax = (gcmax + a.tpc - 1) / a.tpc;
        a.bn_max = 16 * kmax;
        a.bn_small = kmin >= 1 && kmin < kmax ? 16 * kmin : 0;
        a.kblocks = (H + 63) / 64;
        // With at most 64 rows and W tiles of at least 64 rows (8 KB a
        // k-block) the hidden-row box is 64 rows and the stage holds only
        // those: the M = 128 MMA's A rows 64..127 then read the first 8 KB of
        // the same stage's W tile (landed shared memory), which only feeds
        // TMEM lanes of rows >= rows, never read back.  The freed 8 KB a stage
        // buys a deeper ring.  A smaller W tile would leave those 8 KB short
        // of the stage (past the ring's end in the last one), so the A tile
        // then keeps its full 16 KB.
        const bool alias = r <= 64 && a.bn_max >= 64;
        const int h_box = alias ? 64 : 128;
        a.a_bytes = alias ? h_box * 128 : a.mt * LM_A_TILE_BYTES;
        a.stage_bytes = a.a_bytes + a.bn_max * 128;
        a.stages = (SMEM_BUDGET - 2048) / a.stage_bytes;
        if (a.stages > 8) a.stages = 8;
        const int cols = 2 * a.mt * a.bn_max;
        a.tmem_cols = cols <= 32 ? 32 : cols <= 64 ? 64 : cols <= 128 ? 128 : cols <= 256 ? 256 : 512;
        a.mode = mode;
        a.K = K;
        a.logits = logits;
        a.part = part;
        a.err = err;
        CUtensorMap mh, mws, mwb;
        const char* hb = static_cast<const char*>(h) + (size_t)row0 * H * 2;
        int rc = make_map_2d(&mh, hb, (uint64_t)r, (uint64_t)H, (uint32_t)h_box, (uint64_t)H * 2);
        if (rc != GV_OK) return rc;
        rc = make_map_2d(&mwb, W, (uint64_t)V, (uint64_t)H, (uint32_t)a.bn_max, (uint64_t)H * 2);
        if (rc != GV_OK) return rc;
        rc = make_map_2d(&mws, W, (uint64_t)V, (uint64_t)H, (uint32_t)(a.bn_small ? a.bn_small : a.bn_max),
                         (uint64_t)H * 2);
        if (rc != GV_OK) return rc;
        const size_t smem = 1024 + (size_t)a.stages * a.stage_bytes + 8 * (2 * a.stages + 5) + 16;
        if (mode == GV_SELECT_TOPK) {
            cudaFuncSetAttribute(lmhead_tc_kernel<16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem);
            launch_pdl(lmhead_tc_kernel<16>, dim3(grid), dim3(LM_THREADS), smem, st, mh, mws, mwb, a);
        } else {
            cudaFuncSetAttribute(lmhead_tc_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem);
            launch_pdl(lmhead_tc_kernel<1>, dim3(grid), dim3(LM_THREADS), smem, st, mh, mws, mwb, a);
        }
        rc = check_launch("lmhead_tc_kernel");
        if (rc != GV_OK) return rc;
    }
    return GV_OK;
}

}  // namespace gv
