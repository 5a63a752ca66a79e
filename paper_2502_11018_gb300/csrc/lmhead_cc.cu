// gv_lmhead_select, CUDA-core path (fp32 operands) and the selection merge
// shared with the tensor-core path.
//
// GRIFFIN Section 3 / Eq. 1: the LM head maps each node's final hidden state
// to vocabulary scores.  fp32 operands are kept on CUDA cores (FFMA): the
// tensor cores' tf32 mode would round the operands to 10-bit mantissas, well
// outside the 1e-4 relative tolerance fp32 results are held to.
//
// Tile: 64 vocabulary rows x 32 hidden-state rows per 256-thread block, the
// hidden dimension streamed through shared memory 32 at a time; each thread
// owns a 4 (vocab) x 2 (rows) patch of scores.  The selection then runs on
// the tile in shared memory and leaves one partial result per (tile, row) in
// the workspace; lmhead_merge_kernel reduces the partials of every row.
#include "gv_internal.cuh"

namespace gv {

constexpr int CC_TV = 64;   // vocab rows per tile
constexpr int CC_TR = 32;   // hidden-state rows per tile
constexpr int CC_TK = 32;   // hidden dim per stage

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
    __shared__ float sW[CC_TK][CC_TV + 1];
    __shared__ float sH[CC_TK][CC_TR + 1];
    __shared__ float sS[CC_TR][CC_TV + 1];
    const int tid = threadIdx.x;
    const int v0 = blockIdx.x * CC_TV;
    const int r0 = blockIdx.y * CC_TR;
    const int tv = tid & 15, tr = tid >> 4;
    float acc[4][2] = {};
    for (int k0 = 0; k0 < H; k0 += CC_TK) {
        for (int e = tid; e < CC_TV * CC_TK; e += 256) {
            const int vv = e / CC_TK, kk = e % CC_TK;
            const int v = v0 + vv, k = k0 + kk;
            sW[kk][vv] = (v < V && k < H) ? to_f32(W[(size_t)v * H + k]) : 0.f;
        }
        for (int e = tid; e < CC_TR * CC_TK; e += 256) {
            const int rr = e / CC_TK, kk = e % CC_TK;
            const int r = r0 + rr, k = k0 + kk;
            sH[kk][rr] = (r < rows && k < H) ? to_f32(h[(size_t)r * H + k]) : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < CC_TK; ++kk) {
            float wv[4], hv[2];
#pragma unroll
            for (int a = 0; a < 4; ++a) wv[a] = sW[kk][tv + 16 * a];
#pragma unroll
            for (int c = 0; c < 2; ++c) hv[c] = sH[kk][tr + 16 * c];
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int c = 0; c < 2; ++c) acc[a][c] = fmaf(wv[a], hv[c], acc[a][c]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int c = 0; c < 2; ++c) {
            const int vv = tv + 16 * a, rr = tr + 16 * c;
            const bool valid = (v0 + vv < V) && (r0 + rr < rows);
            sS[rr][vv] = valid ? acc[a][c] : -INFINITY;
            if (mode == GV_SELECT_LOGITS && valid) logits[(size_t)(r0 + rr) * V + v0 + vv] = acc[a][c];
        }
    __syncthreads();
    // Selection: warp w handles rows w, w+8, w+16, w+24 of the tile.
    const int warp = tid >> 5, lane = tid & 31;
    const int slot = blockIdx.x;
    for (int rr = warp; rr < CC_TR; rr += 8) {
        const int r = r0 + rr;
        if (r >= rows) break;
        const float x0 = sS[rr][lane], x1 = sS[rr][lane + 32];
        if (mode == GV_SELECT_LOGITS) {
            const float m = warp_max(fmaxf(x0, x1));
            float s = 0.f;
            if (x0 != -INFINITY) s += __expf(x0 - m);
            if (x1 != -INFINITY) s += __expf(x1 - m);
            s = warp_sum(s);
            if (lane == 0) {
                part.m[(size_t)slot * rows + r] = m;
                part.s[(size_t)slot * rows + r] = (m == -INFINITY) ? 0.f : s;
            }
        } else {
            const int i0 = v0 + lane, i1 = v0 + lane + 32;
            const size_t o = ((size_t)slot * rows + r) * K;
            warp_topk(x0, i0 < V ? i0 : INT32_MAX, x1, i1 < V ? i1 : INT32_MAX, K,
                      part.val + o, part.id + o);
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
    if (err != nullptr && *err != 0) {
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
    dim3 grid((V + CC_TV - 1) / CC_TV, (rows + CC_TR - 1) / CC_TR);
    lmhead_cc_kernel<float><<<grid, 256, 0, st>>>(h, W, rows, H, V, mode, K, logits, part);
    const int rc = check_launch("lmhead_cc_kernel");
    if (rc != GV_OK) return rc;
    return launch_lmhead_merge(part, mode, K, ids, vals, row_max, row_lse, nullptr, st);
}

}  // namespace gv
