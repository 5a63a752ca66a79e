// gv_accept: longest accepted root chain of each draft tree.
//
// Greedy (T = 0), GRIFFIN Sections 3/4.1/5: one warp per sequence, two nodes
// per lane.  A match bitmask is formed with ballots (node j matches when its
// token equals the target's choice at its parent); node i is accepted when
// its ancestor mask has no bit outside the match mask; a warp max over
// (depth, -index) picks the deepest accepted node; path slots come from bit
// ranks of that node's ancestor mask.
//
// Sampling (T > 0), Section 5 losslessness with the multi-draft recursive
// rejection rule: one block per sequence walks down the tree.  Each visited
// node costs two passes over the vocabulary for the softmax statistics of the
// target and draft rows, one pass per rejected child for the residual
// max(p - q, 0), and one scan for the final inverse-CDF draw.  Residual
// distributions ping-pong between two fp32 vocabulary rows of the workspace.
#include "gv_internal.cuh"

namespace gv {

__device__ __forceinline__ int parent_of(unsigned long long a, int j) {
    const unsigned long long up = a & ~(1ull << j);
    return up ? 63 - __clzll((long long)up) : -1;
}

__global__ void __launch_bounds__(128)
accept_greedy_kernel(int B, int N, int D, const int32_t* __restrict__ tokens,
                     const unsigned long long* __restrict__ anc, const int32_t* __restrict__ depth,
                     const int32_t* __restrict__ choice, int32_t* __restrict__ path,
                     int32_t* __restrict__ accept_len, int32_t* __restrict__ out_tokens,
                     int32_t* __restrict__ seq_status) {
    pdl_wait();
    pdl_trigger();
    const int b = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (b >= B) return;
    const int W = D + 1;
    const size_t base = (size_t)b * N;
    const bool v0 = lane < N, v1 = lane + 32 < N;
    const unsigned long long a0 = v0 ? anc[base + lane] : 0ull;
    const unsigned long long a1 = v1 ? anc[base + lane + 32] : 0ull;
    const int d0 = v0 ? depth[base + lane] : 0;
    const int d1 = v1 ? depth[base + lane + 32] : 0;
    int st = seq_status[b];
    const bool deep = __any_sync(FULL, (v0 && d0 > D) || (v1 && d1 > D));
    if (st == GV_OK && deep) st = GV_ERR_INVALID_TREE;
    if (st != GV_OK) {
        for (int t = lane; t < W; t += 32) {
            path[(size_t)b * W + t] = -1;
            out_tokens[(size_t)b * W + t] = -1;
        }
        if (lane == 0) {
            accept_len[b] = 0;
            seq_status[b] = st;
        }
        return;
    }
    bool ok0 = true, ok1 = true;
    if (v0 && lane > 0) {
        const int p = parent_of(a0, lane);
        ok0 = p >= 0 && tokens[base + lane] == choice[base + p];
    }
    if (v1) {
        const int p = parent_of(a1, lane + 32);
        ok1 = p >= 0 && tokens[base + lane + 32] == choice[base + p];
    }
    const unsigned long long okmask =
        (unsigned long long)__ballot_sync(FULL, ok0) | ((unsigned long long)__ballot_sync(FULL, ok1) << 32);
    // key = depth * 64 + (63 - index) + 1 for accepted nodes, 0 otherwise.
    unsigned key = 0;
    if (v0 && (a0 & ~okmask) == 0ull) key = (unsigned)d0 * 64u + (63u - lane) + 1u;
    if (v1 && (a1 & ~okmask) == 0ull) key = max(key, (unsigned)d1 * 64u + (31u - lane) + 1u);
    key = __reduce_max_sync(FULL, key);
    const int best = 63 - (int)((key - 1u) & 63u);
    const int bdepth = (int)((key - 1u) >> 6);
    const unsigned long long abest = __shfl_sync(FULL, best < 32 ? a0 : a1, best & 31);
#pragma unroll
    for (int half = 0; half < 2; ++half) {
        const int j = lane + 32 * half;
        if (j < N && ((abest >> j) & 1ull)) {
            const int r = __popcll(abest & ((1ull << j) - 1ull));
            if (r >= W) continue;   // only with an ancestor mask inconsistent with depth
            path[(size_t)b * W + r] = j;
            if (r >= 1) out_tokens[(size_t)b * W + r - 1] = tokens[base + j];
        }
    }
    for (int t = bdepth + 1 + lane; t < W; t += 32) {
        path[(size_t)b * W + t] = -1;
        out_tokens[(size_t)b * W + t] = -1;
    }
    if (lane == 0) {
        out_tokens[(size_t)b * W + bdepth] = choice[base + best];
        accept_len[b] = bdepth + 1;
    }
}

// ---------------------------------------------------------------- sampling --

constexpr int SAMPLE_THREADS = 512;

__device__ float block_reduce(float v, bool is_max, float* red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = is_max ? warp_max(v) : warp_sum(v);
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    if (warp == 0) {
        float x = lane < (int)(blockDim.x >> 5) ? red[lane] : (is_max ? -INFINITY : 0.0f);
        x = is_max ? warp_max(x) : warp_sum(x);
        if (lane == 0) red[32] = x;
    }
    __syncthreads();
    return red[32];
}

__global__ void __launch_bounds__(SAMPLE_THREADS)
accept_sample_kernel(int B, int N, int D, int V, float invT, const int32_t* __restrict__ tokens,
                     const unsigned long long* __restrict__ anc, const int32_t* __restrict__ depth,
                     const float* __restrict__ tlog, const float* __restrict__ dlog,
                     const float* __restrict__ u_acc, const float* __restrict__ u_res,
                     int32_t* __restrict__ path, int32_t* __restrict__ accept_len,
                     int32_t* __restrict__ out_tokens, int32_t* __restrict__ seq_status,
                     float* __restrict__ work) {
    __shared__ int s_par[64];
    __shared__ int s_trail[65];
    __shared__ int s_emit[65];
    __shared__ float red[33];
    __shared__ float s_scan[SAMPLE_THREADS];
    pdl_wait();
    pdl_trigger();
    __shared__ int s_pick;
    const int b = blockIdx.x;
    const int tid = threadIdx.x;
    const int W = D + 1;
    const size_t base = (size_t)b * N;

    int st = seq_status[b];
    int deep = 0, badtok = 0;
    if (tid < N) {
        s_par[tid] = parent_of(anc[base + tid], tid);
        deep = depth[base + tid] > D || (tid > 0 && s_par[tid] < 0);
        const int x = tokens[base + tid];
        badtok = tid > 0 && (x < 0 || x >= V);
    }
    deep = __syncthreads_or(deep);
    badtok = __syncthreads_or(badtok);
    if (st == GV_OK && deep) st = GV_ERR_INVALID_TREE;
    if (st == GV_OK && badtok) st = GV_ERR_ARG;   // a draft token outside [0, V)
    if (st != GV_OK) {
        for (int t = tid; t < W; t += blockDim.x) {
            path[(size_t)b * W + t] = -1;
            out_tokens[(size_t)b * W + t] = -1;
        }
        if (tid == 0) {
            accept_len[b] = 0;
            seq_status[b] = st;
        }
        return;
    }
    float* wbuf[2] = {work + (size_t)b * 2 * V, work + (size_t)b * 2 * V + V};

    int u = 0, len = 0;
    if (tid == 0) s_trail[0] = 0;
    // Each thread owns a contiguous vocabulary segment (for the ordered scan).
    const int seg = (V + blockDim.x - 1) / blockDim.x;
    const int v_lo = min(V, tid * seg), v_hi = min(V, v_lo + seg);
#pragma unroll 1
    // Without draft logits the drafts are deterministic proposals: q(x) = 1
    // for a drafted token, and a rejection zeroes p(x) (q = 0 elsewhere).
    const bool has_q = dlog != nullptr;
    while (true) {
        const float* T = tlog + (base + u) * (size_t)V;
        const float* Q = has_q ? dlog + (base + u) * (size_t)V : nullptr;
        float tm = -INFINITY, qm = -INFINITY;
        for (int v = v_lo; v < v_hi; ++v) {
            tm = fmaxf(tm, T[v] * invT);
            if (has_q) qm = fmaxf(qm, Q[v] * invT);
        }
        tm = block_reduce(tm, true, red);
        if (has_q) qm = block_reduce(qm, true, red);
        float ts = 0.f, qs = 0.f;
        for (int v = v_lo; v < v_hi; ++v) {
            ts += __expf(T[v] * invT - tm);
            if (has_q) qs += __expf(Q[v] * invT - qm);
        }
        ts = block_reduce(ts, false, red);
        if (has_q) qs = block_reduce(qs, false, red);
        const float tinv = 1.0f / ts, qinv = has_q ? 1.0f / qs : 0.f;
        // p(v) = exp(T[v]/T - tm) / ts while mode == 0, else wbuf[cur][v] / wsum.
        int mode = 0, cur = 0;
        float wsum = 1.0f;
        int next = -1;
#pragma unroll 1
        for (int c = u + 1; c < N; ++c) {
            if (s_par[c] != u) continue;
            const int x = tokens[base + c];
            const float px = mode == 0 ? __expf(T[x] * invT - tm) * tinv : wbuf[cur][x] / wsum;
            const float qx = has_q ? __expf(Q[x] * invT - qm) * qinv : 1.0f;
            if (qx == 0.0f || u_acc[base + c] <= px / qx) {
                next = c;
                break;
            }
            float part = 0.f;
            float* dst = wbuf[cur ^ mode];   // first residual goes to buffer 0
            const float winv = 1.0f / wsum;
            for (int v = v_lo; v < v_hi; ++v) {
                const float pv = mode == 0 ? __expf(T[v] * invT - tm) * tinv : wbuf[cur][v] * winv;
                const float r = has_q ? fmaxf(pv - __expf(Q[v] * invT - qm) * qinv, 0.0f) : (v == x ? 0.0f : pv);
                dst[v] = r;
                part += r;
            }
            const float s = block_reduce(part, false, red);
            if (s > 0.0f) {
                cur = cur ^ mode;
                mode = 1;
                wsum = s;
            }
            // s == 0: keep p (buffer `cur` / the softmax) unchanged.
        }
        if (next >= 0) {
            ++len;
            if (tid == 0) {
                s_trail[len] = next;
                s_emit[len - 1] = tokens[base + next];
            }
            u = next;
            __syncthreads();
            continue;
        }
        // Inverse-CDF draw from the current p: segment sums, ordered scan.
        float part = 0.f;
        for (int v = v_lo; v < v_hi; ++v)
            part += mode == 0 ? __expf(T[v] * invT - tm) * tinv : wbuf[cur][v];
        s_scan[tid] = part;
        __syncthreads();
        if (tid == 0) {
            float acc = 0.f;
            for (int t = 0; t < (int)blockDim.x; ++t) {
                const float x = s_scan[t];
                s_scan[t] = acc;
                acc += x;
            }
            red[32] = acc;
            s_pick = -1;
        }
        __syncthreads();
        const float target = u_res[base + u] * red[32];
        float acc = s_scan[tid];
        if (v_lo < v_hi && acc <= target && target < acc + part) {
            int pick = v_hi - 1;
            for (int v = v_lo; v < v_hi; ++v) {
                acc += mode == 0 ? __expf(T[v] * invT - tm) * tinv : wbuf[cur][v];
                if (acc > target) {
                    pick = v;
                    break;
                }
            }
            atomicMax(&s_pick, pick);
        }
        __syncthreads();
        if (tid == 0) {
            int pick = s_pick;
            if (pick < 0) {   // rounding left the target at the very top: last v with p > 0
                for (int v = V - 1; v >= 0; --v) {
                    const float pv = mode == 0 ? __expf(T[v] * invT - tm) * tinv : wbuf[cur][v];
                    if (pv > 0.0f) {
                        pick = v;
                        break;
                    }
                }
                if (pick < 0) pick = 0;
            }
            s_emit[len] = pick;
        }
        __syncthreads();
        break;
    }
    for (int t = tid; t < W; t += blockDim.x) {
        path[(size_t)b * W + t] = t <= len ? s_trail[t] : -1;
        out_tokens[(size_t)b * W + t] = t <= len ? s_emit[t] : -1;
    }
    if (tid == 0) accept_len[b] = len + 1;
}

int launch_accept(int B, int N, int D, int V, float temperature, const int32_t* tokens,
                  const uint64_t* anc, const int32_t* depth, const int32_t* choice,
                  const float* target_logits, const float* draft_logits, const float* u_acc,
                  const float* u_res, int32_t* path, int32_t* accept_len, int32_t* out_tokens,
                  int32_t* seq_status, void* workspace, cudaStream_t st) {
    const auto* a = reinterpret_cast<const unsigned long long*>(anc);
    if (temperature == 0.0f) {
        const int warps_per_block = 4;
        const int blocks = (B + warps_per_block - 1) / warps_per_block;
        launch_pdl(accept_greedy_kernel, dim3(blocks), dim3(32 * warps_per_block), 0, st, B, N, D, tokens,
                   a, depth, choice, path, accept_len, out_tokens, seq_status);
        return check_launch("accept_greedy_kernel");
    }
    launch_pdl(accept_sample_kernel, dim3(B), dim3(SAMPLE_THREADS), 0, st, B, N, D, V, 1.0f / temperature,
               tokens, a, depth, target_logits, draft_logits, u_acc, u_res, path, accept_len, out_tokens,
               seq_status, static_cast<float*>(workspace));
    return check_launch("accept_sample_kernel");
}

}  // namespace gv
