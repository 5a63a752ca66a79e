// gv_lmhead_select, CUDA-core path (fp32 operands) and the selection merge
// shared with the tensor-core path.
//
// GRIFFIN Section 3 / Eq. 1: the LM head maps each node's final hidden state
// to vocabulary scores.  fp32 operands are kept on CUDA cores (FFMA): the
// tensor cores' tf32 mode would round the operands to 10-bit mantissas, well
// outside the 1e-4 relative tolerance fp32 results are held to.
//
// Tile: 16 vocabulary rows x 16 hidden-state rows per 256-thread block
// (grid: vocabulary tiles x row tiles, so a 4096-row vocabulary spreads over
// every SM).  The block stages its W rows and hidden-state rows for 512
// of the hidden dimension at a time in shared memory, every thread's loads in
// flight at once; each thread scores a 2 x 4 sub-tile (vocabulary rows
// vq + 8 i against hidden-state rows rq + 4 j: 8 accumulators, 6 16-byte
// shared-memory loads per 32 FMAs), and the 8 warps take interleaved 4-wide
// slices of the hidden dimension, summed across warps at the end.  The selection then
// runs on the tile in shared memory and leaves one partial result per (tile,
// row) in the workspace; lmhead_merge_kernel reduces the partials of every
// row.
#include "gv_internal.cuh"

namespace gv {

constexpr int CC_TV = 16;            // vocab rows per tile (a multiple of 8, at most a warp's lanes)
constexpr int CC_VI = CC_TV / 8;      // vocabulary rows per thread
constexpr int CC_TR = 16;            // hidden-state rows per tile
constexpr int CC_KC = 512;           // hidden dim staged per pass
constexpr int CC_KS = CC_KC + 4;     // staged row stride: 16-byte rows, the 8 lanes of a
                                     // quarter-warp's 16-byte loads on distinct banks
constexpr size_t CC_SMEM = sizeof(float) * ((size_t)(CC_TV + CC_TR) * CC_KS + 8 * CC_TR * (CC_TV + 1) +
                                            CC_TR * (CC_TV + 1));

// Top-K (value desc, id asc) of `cnt` candidates held two per lane, by K
// rounds of warp argmax.  Lane 0 returns the lists.
__device__ void warp_topk(float v0, int i0, float v1, int i1, int K, float* out_v, int* out_i) {
    for (int r = 0; r < K; ++r) {
        float bv = v0;
        int bi = i0;
        if (better(v1, i1, bv, bi)) {
            bv = v1;
            bi = i1;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ov = __shfl_xor_sync(FULL, bv, o);
            const int oi = __shfl_xor_sync(FULL, bi, o);
            if (better(ov, oi, bv, bi)) {
                bv = ov;
                bi = oi;
            }
        }
        if ((threadIdx.x & 31) == 0) {
            out_v[r] = bv;
            out_i[r] = bi;
        }
        if (i0 == bi) {
            v0 = -INFINITY;
            i0 = INT32_MAX;
        }
        if (i1 == bi) {
            v1 = -INFINITY;
            i1 = INT32_MAX;
        }
    }
}

template <typename T>
__global__ void __launch_bounds__(256)
lmhead_cc_kernel(const T* __restrict__ h, const T* __restrict__ W, int rows, int H, int V,
                 int mode, int K, float* __restrict__ logits, SelectPartials part) {
    static_assert(sizeof(T) == 4, "the CUDA-core LM head stages fp32 operands");
    extern __shared__ float cc_smem[];
    float* sW = cc_smem;                              // [CC_TV][CC_KS]
    float* sH = sW + CC_TV * CC_KS;                   // [CC_TR][CC_KS]
    float* sRed = sH + CC_TR * CC_KS;                 // [8 warps][CC_TR][CC_TV + 1]
    float(*sS)[CC_TV + 1] = reinterpret_cast<float(*)[CC_TV + 1]>(sRed + 8 * CC_TR * (CC_TV + 1));
    pdl_wait();
    pdl_trigger();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int v0 = blockIdx.x * CC_TV;
    const int r0 = blockIdx.y * CC_TR;
    // Thread (warp w, lane): vocabulary rows vq + 8 i and hidden rows
    // rq + 4 j (i, j < 4) of the tile, hidden dimension 4 w, 4 w + 32, ...
    const int vq = lane & 7, rq = lane >> 3;
    float acc[CC_VI][4];
#pragma unroll
    for (int i = 0; i < CC_VI; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
    for (int k0 = 0; k0 < H; k0 += CC_KC) {
        const int kc = min(CC_KC, H - k0), kc4 = (kc + 3) & ~3;
        __syncthreads();
        // Stage W rows v0.. and hidden rows r0.. for k0 .. k0 + kc (zeros past
        // the vocabulary, the rows and kc, up to kc4).
        if ((H & 3) == 0) {
            // 16-byte rows: float4 loads (kc is then a multiple of 4), each
            // thread's loads issued together before its stores.
            const int q4 = kc >> 2;
            constexpr int NW = CC_TV * (CC_KC / 4) / 256, NH = CC_TR * (CC_KC / 4) / 256;
            float4 xw[NW], xh[NH];
#pragma unroll
            for (int i = 0; i < NW; ++i) {
                const int e = tid + 256 * i, vv = e / q4, kk = 4 * (e - vv * q4), v = v0 + vv;
                xw[i] = (vv < CC_TV && v < V) ? *reinterpret_cast<const float4*>(W + (size_t)v * H + k0 + kk)
                                              : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int i = 0; i < NH; ++i) {
                const int e = tid + 256 * i, rr = e / q4, kk = 4 * (e - rr * q4), r = r0 + rr;
                xh[i] = (rr < CC_TR && r < rows) ? *reinterpret_cast<const float4*>(h + (size_t)r * H + k0 + kk)
                                                 : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int i = 0; i < NW; ++i) {
                const int e = tid + 256 * i, vv = e / q4, kk = 4 * (e - vv * q4);
                if (vv < CC_TV) *reinterpret_cast<float4*>(sW + vv * CC_KS + kk) = xw[i];
            }
#pragma unroll
            for (int i = 0; i < NH; ++i) {
                const int e = tid + 256 * i, rr = e / q4, kk = 4 * (e - rr * q4);
                if (rr < CC_TR) *reinterpret_cast<float4*>(sH + rr * CC_KS + kk) = xh[i];
            }
        } else {
            for (int e = tid; e < CC_TV * kc4; e += 256) {
                const int vv = e / kc4, kk = e - vv * kc4;
                const int v = v0 + vv;
                sW[vv * CC_KS + kk] = (v < V && kk < kc) ? to_f32(W[(size_t)v * H + k0 + kk]) : 0.f;
            }
            for (int e = tid; e < CC_TR * kc4; e += 256) {
                const int rr = e / kc4, kk = e - rr * kc4;
                const int r = r0 + rr;
                sH[rr * CC_KS + kk] = (r < rows && kk < kc) ? to_f32(h[(size_t)r * H + k0 + kk]) : 0.f;
            }
        }
        __syncthreads();
        // (a warp's 16-byte loads hit 8 consecutive W rows and 4 consecutive
        // hidden rows, each shared by 4 or 8 lanes: distinct bank groups)
        for (int kk = 4 * warp; kk < kc4; kk += 32) {
            float4 w4[CC_VI], h4[4];
#pragma unroll
            for (int i = 0; i < CC_VI; ++i) w4[i] = *reinterpret_cast<const float4*>(sW + (vq + 8 * i) * CC_KS + kk);
#pragma unroll
            for (int j = 0; j < 4; ++j) h4[j] = *reinterpret_cast<const float4*>(sH + (rq + 4 * j) * CC_KS + kk);
#pragma unroll
            for (int i = 0; i < CC_VI; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    acc[i][j] = fmaf(w4[i].x, h4[j].x,
                                     fmaf(w4[i].y, h4[j].y, fmaf(w4[i].z, h4[j].z, fmaf(w4[i].w, h4[j].w, acc[i][j]))));
        }
    }
    // Sum the warps' slices of the hidden dimension.
#pragma unroll
    for (int i = 0; i < CC_VI; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) sRed[(warp * CC_TR + rq + 4 * j) * (CC_TV + 1) + vq + 8 * i] = acc[i][j];
    __syncthreads();
    for (int e = tid; e < CC_TR * CC_TV; e += 256) {
        const int rr = e / CC_TV, vv = e % CC_TV;
        float x = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w) x += sRed[(w * CC_TR + rr) * (CC_TV + 1) + vv];
        const bool valid = (v0 + vv < V) && (r0 + rr < rows);
        sS[rr][vv] = valid ? x : -INFINITY;
        if (mode == GV_SELECT_LOGITS && valid) logits[(size_t)(r0 + rr) * V + v0 + vv] = x;
    }
    __syncthreads();
    // Selection: warp w handles rows w and w + 8 of the tile, lane l the
    // tile's vocabulary row l.
    const int slot = blockIdx.x;
    for (int rr = warp; rr < CC_TR; rr += 8) {
        const int r = r0 + rr;
        if (r >= rows) break;
        const float x0 = lane < CC_TV ? sS[rr][lane] : -INFINITY;
        if (mode == GV_SELECT_LOGITS) {
            const float m = warp_max(x0);
            float s = 0.f;
            if (x0 != -INFINITY) s += __expf(x0 - m);
            s = warp_sum(s);
            if (lane == 0) {
                part.m[(size_t)slot * rows + r] = m;
                part.s[(size_t)slot * rows + r] = (m == -INFINITY) ? 0.f : s;
            }
        } else {
            const int i0 = v0 + lane;
            const size_t o = ((size_t)slot * rows + r) * K;
            warp_topk(x0, i0 < V ? i0 : INT32_MAX, -INFINITY, INT32_MAX, K, part.val + o, part.id + o);
        }
    }
}

// One block per row: merge the per-slot partial lists of that row.
__global__ void __launch_bounds__(256)
lmhead_merge_kernel(SelectPartials part, int mode, int K, int32_t* __restrict__ ids,
                    float* __restrict__ vals, float* __restrict__ row_max,
                    float* __restrict__ row_lse, const int* __restrict__ err) {
    __shared__ float sv[8][16];
    __shared__ int si[8][16];
    __shared__ float red[33];
    pdl_wait();
    pdl_trigger();
    const int r = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int rows = part.rows;
    // err: the projection kernel's per-CTA status words (one per slot)
    if (err != nullptr && __syncthreads_or(tid < part.slots && err[tid] != 0)) {
        // A bounded wait in the projection kernel gave up: no valid result.
        if (mode == GV_SELECT_LOGITS) {
            if (tid == 0 && row_max) row_max[r] = NAN;
            if (tid == 0 && row_lse) row_lse[r] = NAN;
        } else if (tid < K) {
            ids[(size_t)r * K + tid] = -1;
            if (vals) vals[(size_t)r * K + tid] = NAN;
        }
        return;
    }
    if (mode == GV_SELECT_LOGITS) {
        float m = -INFINITY;
        for (int s = tid; s < part.slots; s += blockDim.x) m = fmaxf(m, part.m[(size_t)s * rows + r]);
        m = warp_max(m);
        if (lane == 0) red[warp] = m;
        __syncthreads();
        if (tid == 0) {
            float x = -INFINITY;
            for (int w = 0; w < (int)(blockDim.x >> 5); ++w) x = fmaxf(x, red[w]);
            red[32] = x;
        }
        __syncthreads();
        const float M = red[32];
        float s = 0.f;
        for (int t = tid; t < part.slots; t += blockDim.x) {
            const float pm = part.m[(size_t)t * rows + r];
            if (pm != -INFINITY) s += part.s[(size_t)t * rows + r] * __expf(pm - M);
        }
        s = warp_sum(s);
        __syncthreads();
        if (lane == 0) red[warp] = s;
        __syncthreads();
        if (tid == 0) {
            float x = 0.f;
            for (int w = 0; w < (int)(blockDim.x >> 5); ++w) x += red[w];
            if (row_max) row_max[r] = M;
            if (row_lse) row_lse[r] = M + logf(x);
        }
        return;
    }
    // Top-K over all slots' candidates: K rounds; round q picks, block-wide,
    // the best candidate that comes strictly after pick q-1 in the order
    // (value desc, id asc).  Ids are unique across slots (disjoint vocabulary
    // tiles), so the order is total and no candidate is picked twice.
    const int n = part.slots * K;
    float pv = INFINITY;
    int pi = -1;
    for (int q = 0; q < K; ++q) {
        float bv = -INFINITY;
        int bi = INT32_MAX;
        for (int e = tid; e < n; e += blockDim.x) {
            const int s = e / K, j = e % K;
            const size_t o = ((size_t)s * rows + r) * K + j;
            const int ci = part.id[o];
            if (ci == INT32_MAX) continue;
            float cv = part.val[o];
            if (cv != cv) cv = -INFINITY;
            if (better(pv, pi, cv, ci) && better(cv, ci, bv, bi)) {
                bv = cv;
                bi = ci;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ov = __shfl_xor_sync(FULL, bv, o);
            const int oi = __shfl_xor_sync(FULL, bi, o);
            if (better(ov, oi, bv, bi)) {
                bv = ov;
                bi = oi;
            }
        }
        __syncthreads();
        if (lane == 0) {
            sv[warp][0] = bv;
            si[warp][0] = bi;
        }
        __syncthreads();
        if (tid == 0) {
            for (int w = 1; w < (int)(blockDim.x >> 5); ++w)
                if (better(sv[w][0], si[w][0], bv, bi)) {
                    bv = sv[w][0];
                    bi = si[w][0];
                }
            sv[0][1] = bv;
            si[0][1] = bi;
            ids[(size_t)r * K + q] = bi == INT32_MAX ? -1 : bi;
            if (vals) vals[(size_t)r * K + q] = bv;
        }
        __syncthreads();
        pv = sv[0][1];
        pi = si[0][1];
    }
}

int launch_lmhead_merge(SelectPartials part, int mode, int K, int32_t* ids, float* vals,
                        float* row_max, float* row_lse, const int* err, cudaStream_t st) {
    launch_pdl(lmhead_merge_kernel, dim3(part.rows), dim3(256), 0, st, part, mode, K, ids, vals, row_max,
               row_lse, err);
    return check_launch("lmhead_merge_kernel");
}

int launch_lmhead_cc(const float* h, const float* W, int rows, int H, int V, int mode, int K,
                     float* logits, SelectPartials part, int32_t* ids, float* vals, float* row_max,
                     float* row_lse, cudaStream_t st) {
    static thread_local int attr_dev = -1;
    int dev = 0;
    cudaGetDevice(&dev);
    if (attr_dev != dev) {
        cudaFuncSetAttribute(lmhead_cc_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)CC_SMEM);
        attr_dev = dev;
    }
    dim3 grid((V + CC_TV - 1) / CC_TV, (rows + CC_TR - 1) / CC_TR);
    launch_pdl(lmhead_cc_kernel<float>, grid, dim3(256), CC_SMEM, st, h, W, rows, H, V, mode, K, logits, part);
    const int rc = check_launch("lmhead_cc_kernel");
    if (rc != GV_OK) return rc;
    return launch_lmhead_merge(part, mode, K, ids, vals, row_max, row_lse, nullptr, st);
}

}  // namespace gv
