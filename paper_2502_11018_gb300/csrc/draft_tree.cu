// gv_draft_tree_*: the dynamic draft tree of one GRIFFIN cycle, built from
// top-k expansions and a final rerank (the EAGLE-2 construction the paper's
// Implementation Details appendix uses: 60 nodes, depth 6).
//
// Per sequence, a pool of nodes (token, parent, score) lives in the
// workspace: the root (score 0) and, per expansion step j, the k best tokens
// of each expanded node's draft distribution, scored parent score + log
// softmax.  The k best candidates of step j are the nodes expanded at step
// j + 1 (their slots, best first, index the next step's logits); the rerank
// keeps the N - 1 best pool nodes and the root, in pool order.  Orderings:
// larger score first, then the earlier pool position; within a row, larger
// logit first, then the lower token id.  fp32 throughout.
//
// Kernels: draft_topk_kernel splits each logit row over S CTAs (a partial
// top-k and a partial (max, sum exp) per CTA); draft_select_kernel (one CTA
// per sequence) merges them into each row's top-k and log-sum-exp, appends
// the candidates and picks the next step's expanded nodes;
// draft_rerank_kernel (one CTA per sequence) sorts the pool by score and
// writes the tree.
#include <climits>

#include "gv_internal.cuh"

namespace gv {

constexpr int DT_THREADS = 256;
constexpr int DT_KMAX = 16;
constexpr int DT_SEL_THREADS = 512;          // 16 warps: one per expanded row
constexpr int DT_RR_THREADS = 1024;
constexpr int DT_PMAX = 4096;                // pool capacity of the rerank sort

struct TreeWs {
    int32_t* token;      // [B][P]
    int32_t* parent;     // [B][P]
    float* score;        // [B][P]
    int32_t* exp_id;     // [B][k]  pool ids of the nodes being expanded, best first
    float* pv;           // [B][k][S][k] partial top-k values
    int32_t* pi;         // [B][k][S][k] partial top-k ids
    float* pm;           // [B][k][S] partial max
    float* ps;           // [B][k][S] partial sum of exp(x - max)
};

__host__ __device__ inline int tree_pool_size(int k, int D) { return 1 + k + (D - 1) * k * k; }
__host__ __device__ inline int tree_pool_off(int k, int step) { return step == 0 ? 1 : 1 + k + (step - 1) * k * k; }

static int tree_splits(int V) {
    int s = (V + 4095) / 4096;
    return s < 1 ? 1 : s > 32 ? 32 : s;
}

static size_t al256(size_t x) { return (x + 255) & ~(size_t)255; }

static size_t tree_ws_layout(int B, int k, int D, int V, uint8_t* base, TreeWs* w) {
    const int P = tree_pool_size(k, D), S = tree_splits(V);
    size_t off = 0;
    auto take = [&](size_t bytes) {
        uint8_t* p = base ? base + off : nullptr;
        off += al256(bytes);
        return p;
    };
    TreeWs t;
    t.token = reinterpret_cast<int32_t*>(take((size_t)B * P * 4));
    t.parent = reinterpret_cast<int32_t*>(take((size_t)B * P * 4));
    t.score = reinterpret_cast<float*>(take((size_t)B * P * 4));
    t.exp_id = reinterpret_cast<int32_t*>(take((size_t)B * k * 4));
    t.pv = reinterpret_cast<float*>(take((size_t)B * k * S * k * 4));
    t.pi = reinterpret_cast<int32_t*>(take((size_t)B * k * S * k * 4));
    t.pm = reinterpret_cast<float*>(take((size_t)B * k * S * 4));
    t.ps = reinterpret_cast<float*>(take((size_t)B * k * S * 4));
    if (w) *w = t;
    return off;
}

size_t draft_tree_workspace_bytes(int B, int k, int D, int V) { return tree_ws_layout(B, k, D, V, nullptr, nullptr); }

__device__ __forceinline__ float ld_logit(const float* p) { return *p; }
__device__ __forceinline__ float ld_logit(const __nv_bfloat16* p) { return __bfloat162float(*p); }

// (m, s) pairs of a log-sum-exp: s = sum exp(x - m).
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
    if (m2 > m) {
        s = s * expf(m - m2) + s2;
        m = m2;
    } else if (m2 > -INFINITY) {
        s += s2 * expf(m2 - m);
    }
}

// (value, id) order of every selection here: larger value first, then the
// lower id.
__device__ __forceinline__ bool dt_better(float va, int ia, float vb, int ib) {
    return va > vb || (va == vb && ia < ib);
}

// The warp-wide best of one (value, id, tag) per lane; every lane gets it
// (ids are unique among real entries; placeholders are (-inf, INT_MAX)).
__device__ __forceinline__ void warp_best(float& v, int& id, int& tag) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float v2 = __shfl_xor_sync(FULL, v, o);
        const int i2 = __shfl_xor_sync(FULL, id, o), t2 = __shfl_xor_sync(FULL, tag, o);
        if (dt_better(v2, i2, v, id)) {
            v = v2;
            id = i2;
            tag = t2;
        }
    }
}

// One CTA per (row, split) of DT_ITEMS values a thread at most: the split's
// top-k and its (max, sum exp).  Each warp bounds its top-k from below by the
// k-th largest of its lanes' maxima (those k maxima are k of its values), so
// only values at or above that bound are ranked: they are compacted into a
// shared buffer (a fallback ranks all of the warp's values when more than
// DT_CAP pass) and the warp extracts its k best; warp 0 then merges the
// warps' lists.
constexpr int DT_ITEMS_MAX = 32;             // a split holds at most 8192 values
constexpr int DT_CAP = 64;                   // compacted candidates per warp
constexpr int DT_WARPS = DT_THREADS / 32;

template <typename T, int DT_ITEMS>
__global__ void __launch_bounds__(DT_THREADS)
draft_topk_kernel(const T* __restrict__ logits, int rows, int V, int S, int k, TreeWs w) {
    __shared__ float cv[DT_WARPS][DT_CAP];
    __shared__ int ci[DT_WARPS][DT_CAP];
    __shared__ float wlv[DT_WARPS * DT_KMAX];
    __shared__ int wli[DT_WARPS * DT_KMAX];
    __shared__ float rm[DT_WARPS], rs[DT_WARPS];
    pdl_wait();
    pdl_trigger();
    const int row = blockIdx.x / S, sp = blockIdx.x % S;          // row = b * rows + r
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int c0 = (int)(((long)V * sp) / S), c1 = (int)(((long)V * (sp + 1)) / S);
    const T* x = logits + (size_t)row * V;
    float vals[DT_ITEMS];
#pragma unroll
    for (int u = 0; u < DT_ITEMS; ++u) {
        const int v = c0 + u * DT_THREADS + tid;
        vals[u] = v < c1 ? ld_logit(x + v) : -INFINITY;
    }
    float lm = -INFINITY;
#pragma unroll
    for (int u = 0; u < DT_ITEMS; ++u) lm = fmaxf(lm, vals[u]);
    float ls = 0.f;
    if (lm > -INFINITY) {
#pragma unroll
        for (int u = 0; u < DT_ITEMS; ++u) ls += expf(vals[u] - lm);    // exp(-inf) = 0 for the padding
    }
    // the k-th largest lane maximum: bitonic sort of the lanes' maxima, descending
    float sv = lm;
#pragma unroll
    for (int size = 2; size <= 32; size <<= 1)
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            const float o = __shfl_xor_sync(FULL, sv, stride);
            const bool desc = (lane & size) == 0, lower = (lane & stride) == 0;
            sv = (lower == desc) ? fmaxf(sv, o) : fminf(sv, o);
        }
    const float thr = __shfl_sync(FULL, sv, k - 1);
    // compact the values >= thr (the ballots first, then their running offsets)
    unsigned bal[DT_ITEMS];
#pragma unroll
    for (int u = 0; u < DT_ITEMS; ++u) bal[u] = __ballot_sync(FULL, c0 + u * DT_THREADS + tid < c1 && vals[u] >= thr);
    int cnt = 0;
    const unsigned below = (1u << lane) - 1u;
#pragma unroll
    for (int u = 0; u < DT_ITEMS; ++u) {
        const int pos = cnt + __popc(bal[u] & below);
        if (((bal[u] >> lane) & 1u) && pos < DT_CAP) {
            cv[warp][pos] = vals[u];
            ci[warp][pos] = c0 + u * DT_THREADS + tid;
        }
        cnt += __popc(bal[u]);
    }
    __syncwarp();
    if (cnt <= DT_CAP) {
        // each candidate's place among the warp's candidates, by counting the
        // better ones; the first k places form the warp's list
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int c = lane + 32 * h;
            if (c < cnt) {
                const float a = cv[warp][c];
                const int ai = ci[warp][c];
                int rank = 0;
                for (int q = 0; q < cnt; ++q) rank += dt_better(cv[warp][q], ci[warp][q], a, ai) ? 1 : 0;
                if (rank < k) {
                    wlv[warp * DT_KMAX + rank] = a;
                    wli[warp * DT_KMAX + rank] = ai;
                }
            }
        }
        // fewer than k candidates (a warp with fewer than k values): pad
        for (int q = cnt + lane; q < k; q += 32) {
            wlv[warp * DT_KMAX + q] = -INFINITY;
            wli[warp * DT_KMAX + q] = INT_MAX;
        }
    } else {
        // many values tie at the bound: rank all of the warp's values
        uint32_t taken = 0;
        for (int j = 0; j < k; ++j) {
            float bv = -INFINITY;
            int bi = INT_MAX, bu = 0;
#pragma unroll
            for (int u = 0; u < DT_ITEMS; ++u) {
                const int v = c0 + u * DT_THREADS + tid;
                if (v < c1 && !(taken & (1u << u)) && dt_better(vals[u], v, bv, bi)) {
                    bv = vals[u];
                    bi = v;
                    bu = u;
                }
            }
            int bl = lane;
            warp_best(bv, bi, bl);
            if (lane == bl) taken |= 1u << bu;      // (bu is this lane's own)
            if (lane == 0) {
                wlv[warp * DT_KMAX + j] = bv;
                wli[warp * DT_KMAX + j] = bi;
            }
        }
    }
    // (max, sum exp) over the CTA
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(FULL, lm, o), s2 = __shfl_xor_sync(FULL, ls, o);
        lse_merge(lm, ls, m2, s2);
    }
    if (lane == 0) {
        rm[warp] = lm;
        rs[warp] = ls;
    }
    __syncthreads();
    if (warp != 0) return;
    const size_t pbase = (size_t)row * S + sp;
    if (lane == 0) {
        float M = rm[0], Ssum = rs[0];
        for (int q = 1; q < DT_WARPS; ++q) lse_merge(M, Ssum, rm[q], rs[q]);
        w.pm[pbase] = M;
        w.ps[pbase] = Ssum;
    }
    // merge the warps' sorted lists: the CTA's k best are at or above the
    // largest of the warps' k-th values (that warp alone has k such entries);
    // compact those entries and place each by counting the better ones
    float kth = -INFINITY;
    if (lane < DT_WARPS) kth = wlv[lane * DT_KMAX + k - 1];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) kth = fmaxf(kth, __shfl_xor_sync(FULL, kth, o));
    const int tot = DT_WARPS * k;
    float* mv = &cv[0][0];                    // every warp's buffer is free now: DT_WARPS * DT_CAP >= tot
    int* mi = &ci[0][0];
    int n = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int t = lane + 32 * q;
        const int src = t < tot ? (t / k) * DT_KMAX + t % k : 0;
        const float a = t < tot ? wlv[src] : -INFINITY;
        const int ai = t < tot ? wli[src] : INT_MAX;
        const bool p = ai != INT_MAX && a >= kth;
        const unsigned bq = __ballot_sync(FULL, p);
        if (p) {
            const int pos = n + __popc(bq & ((1u << lane) - 1u));
            mv[pos] = a;
            mi[pos] = ai;
        }
        n += __popc(bq);
    }
    __syncwarp();
    for (int c = lane; c < n; c += 32) {
        const float a = mv[c];
        const int ai = mi[c];
        int rank = 0;
        for (int q = 0; q < n; ++q) rank += dt_better(mv[q], mi[q], a, ai) ? 1 : 0;
        if (rank < k) {
            w.pv[pbase * k + rank] = a;
            w.pi[pbase * k + rank] = ai;
        }
    }
}

// One CTA per sequence: each row's top-k and log-sum-exp from its splits
// (warp r merges row r), the candidates appended to the pool, and the next
// step's expanded nodes.
__global__ void __launch_bounds__(DT_SEL_THREADS)
draft_select_kernel(int rows, int S, int k, int D, int step, const int32_t* __restrict__ root_token, TreeWs w,
                    int32_t* __restrict__ exp_token, int32_t* __restrict__ exp_pool) {
    __shared__ float cs[DT_KMAX * DT_KMAX];
    __shared__ int ct[DT_KMAX * DT_KMAX];
    pdl_wait();
    pdl_trigger();
    const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int P = tree_pool_size(k, D), off = tree_pool_off(k, step);
    int32_t* tok = w.token + (size_t)b * P;
    int32_t* par = w.parent + (size_t)b * P;
    float* sc = w.score + (size_t)b * P;
    if (step == 0 && tid == 0) {
        tok[0] = root_token[b];
        par[0] = -1;
        sc[0] = 0.f;
    }
    if (warp < rows) {
        const int r = warp;
        const int pid = step == 0 ? 0 : w.exp_id[b * k + r];
        const float base = step == 0 ? 0.f : sc[pid];
        const size_t rb = ((size_t)b * rows + r) * S;
        float m = lane < S ? w.pm[rb + lane] : -INFINITY;
        float s = lane < S ? w.ps[rb + lane] : 0.f;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float m2 = __shfl_xor_sync(FULL, m, o), s2 = __shfl_xor_sync(FULL, s, o);
            lse_merge(m, s, m2, s2);
        }
        const float lse = m + logf(s);
        // this lane's split list in registers (all loads issued at once);
        // a round's winner shifts its list up by one
        float lv[DT_KMAX];
        int li[DT_KMAX];
#pragma unroll
        for (int q = 0; q < DT_KMAX; ++q) {
            const bool ok = lane < S && q < k;
            lv[q] = ok ? w.pv[(rb + lane) * k + q] : -INFINITY;
            li[q] = ok ? w.pi[(rb + lane) * k + q] : INT_MAX;
        }
        for (int j = 0; j < k; ++j) {
            float bv = lv[0];
            int bi = li[0];
            int bl = lane;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const float v2 = __shfl_xor_sync(FULL, bv, o);
                const int i2 = __shfl_xor_sync(FULL, bi, o), l2 = __shfl_xor_sync(FULL, bl, o);
                if (v2 > bv || (v2 == bv && i2 < bi)) {
                    bv = v2;
                    bi = i2;
                    bl = l2;
                }
            }
            if (lane == bl) {
#pragma unroll
                for (int q = 0; q + 1 < DT_KMAX; ++q) {
                    lv[q] = lv[q + 1];
                    li[q] = li[q + 1];
                }
                lv[DT_KMAX - 1] = -INFINITY;
                li[DT_KMAX - 1] = INT_MAX;
            }
            if (lane == 0) {
                const int c = r * k + j;
                const float score = base + (bv - lse);
                tok[off + c] = bi;
                par[off + c] = pid;
                sc[off + c] = score;
                cs[c] = score != score ? -INFINITY : score;     // NaN never wins
                ct[c] = bi;
            }
        }
    }
    if (step + 1 >= D) return;
    __syncthreads();
    // the k best candidates (larger score, then the earlier pool position):
    // a candidate's place is the number of better ones
    const int nc = rows * k;
    if (tid < nc) {
        const float a = cs[tid];
        int rank = 0;
        for (int q = 0; q < nc; ++q) rank += dt_better(cs[q], q, a, tid) ? 1 : 0;
        if (rank < k) {
            const int id = off + tid;
            w.exp_id[b * k + rank] = id;
            if (exp_pool) exp_pool[b * k + rank] = id;
            if (exp_token) exp_token[b * k + rank] = ct[tid];
        }
    }
}

// Sort key: ascending key = descending score, then ascending pool id.  NaN
// scores sort last.
__device__ __forceinline__ unsigned long long rank_key(float score, int id) {
    if (score != score) score = -INFINITY;
    uint32_t u = __float_as_uint(score);
    u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);      // ascending with the float
    return ((unsigned long long)(~u) << 32) | (uint32_t)id;
}

// One CTA per sequence: bitonic sort of the pool (root excluded) by rank_key,
// keep the first N - 1 and the root, number them in pool order, and write the
// tree (parents remapped to tree indices).
__global__ void __launch_bounds__(DT_RR_THREADS)
draft_rerank_kernel(int k, int D, int N, TreeWs w, int32_t* __restrict__ parents, int32_t* __restrict__ tokens) {
    __shared__ unsigned long long key[DT_PMAX];
    __shared__ int16_t newidx[DT_PMAX];          // pool position -> tree index, -1 if dropped
    pdl_wait();
    pdl_trigger();
    const int b = blockIdx.x, tid = threadIdx.x;
    const int P = tree_pool_size(k, D);
    const int32_t* tok = w.token + (size_t)b * P;
    const int32_t* par = w.parent + (size_t)b * P;
    const float* sc = w.score + (size_t)b * P;
    int n2 = 1;
    while (n2 < P - 1) n2 <<= 1;
    for (int i = tid; i < n2; i += DT_RR_THREADS)
        key[i] = i < P - 1 ? rank_key(sc[i + 1], i + 1) : ~0ull;
    for (int i = tid; i < P; i += DT_RR_THREADS) newidx[i] = 0;
    __syncthreads();
    for (int size = 2; size <= n2; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int i = tid; i < n2; i += DT_RR_THREADS) {
                const int j = i ^ stride;
                if (j > i) {
                    const bool up = (i & size) == 0;
                    const unsigned long long a = key[i], c = key[j];
                    if ((a > c) == up) {
                        key[i] = c;
                        key[j] = a;
                    }
                }
            }
            __syncthreads();
        }
    // kept flags (the root and the first N - 1 keys), then tree indices in
    // pool order: each thread numbers DT_PMAX / DT_RR_THREADS consecutive
    // entries after an exclusive scan of the per-thread counts
    __shared__ int wsum[DT_RR_THREADS / 32];
    for (int i = tid; i < N - 1; i += DT_RR_THREADS) newidx[(int)(key[i] & 0xffffffffu)] = 1;
    if (tid == 0) newidx[0] = 1;
    __syncthreads();
    constexpr int PER = DT_PMAX / DT_RR_THREADS;
    int cnt = 0;
#pragma unroll
    for (int q = 0; q < PER; ++q) {
        const int i = tid * PER + q;
        cnt += (i < P && newidx[i]) ? 1 : 0;
    }
    const int lane = tid & 31, warp = tid >> 5;
    int incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(FULL, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    int before = 0;
    for (int q = 0; q < warp; ++q) before += wsum[q];
    int c = before + incl - cnt;
#pragma unroll
    for (int q = 0; q < PER; ++q) {
        const int i = tid * PER + q;
        if (i < P) newidx[i] = (int16_t)(newidx[i] ? c++ : -1);
    }
    __syncthreads();
    for (int i = tid; i < P; i += DT_RR_THREADS) {
        const int t = newidx[i];
        if (t < 0) continue;
        tokens[(size_t)b * N + t] = tok[i];
        parents[(size_t)b * N + t] = i == 0 ? -1 : newidx[par[i]];
    }
}

int launch_draft_tree_expand(int B, int k, int D, int V, int step, int dt, const int32_t* root_token,
                             const void* logits, int32_t* exp_token, int32_t* exp_pool, void* ws, cudaStream_t st) {
    TreeWs w;
    tree_ws_layout(B, k, D, V, static_cast<uint8_t*>(ws), &w);
    const int rows = step == 0 ? 1 : k, S = tree_splits(V);
    const dim3 grid((unsigned)(B * rows * S));
    // values a thread holds: the largest split (ceil(V / S)) over the CTA's threads
    const int chunk = (V + S - 1) / S;
    const bool small = chunk <= 16 * DT_THREADS;
    if (dt == GV_F32) {
        const float* lg = static_cast<const float*>(logits);
        if (small)
            launch_pdl(draft_topk_kernel<float, 16>, grid, dim3(DT_THREADS), 0, st, lg, rows, V, S, k, w);
        else
            launch_pdl(draft_topk_kernel<float, DT_ITEMS_MAX>, grid, dim3(DT_THREADS), 0, st, lg, rows, V, S, k, w);
    } else {
        const __nv_bfloat16* lg = static_cast<const __nv_bfloat16*>(logits);
        if (small)
            launch_pdl(draft_topk_kernel<__nv_bfloat16, 16>, grid, dim3(DT_THREADS), 0, st, lg, rows, V, S, k, w);
        else
            launch_pdl(draft_topk_kernel<__nv_bfloat16, DT_ITEMS_MAX>, grid, dim3(DT_THREADS), 0, st, lg, rows, V, S,
                       k, w);
    }
    int rc = check_launch("draft_topk_kernel");
    if (rc != GV_OK) return rc;
    launch_pdl(draft_select_kernel, dim3(B), dim3(DT_SEL_THREADS), 0, st, rows, S, k, D, step, root_token, w,
               exp_token, exp_pool);
    return check_launch("draft_select_kernel");
}

int launch_draft_tree_finish(int B, int k, int D, int N, int32_t* parents, int32_t* tokens, void* ws,
                             cudaStream_t st) {
    TreeWs w;
    tree_ws_layout(B, k, D, 1, static_cast<uint8_t*>(ws), &w);
    launch_pdl(draft_rerank_kernel, dim3(B), dim3(DT_RR_THREADS), 0, st, k, D, N, w, parents, tokens);
    return check_launch("draft_rerank_kernel");
}

}  // namespace gv
