// gv_kv_compact: append the accepted root chain's K/V rows to every layer's
// cache (GRIFFIN Section 4.1: only the accepted chain survives verification).
//
// One thread per 16-byte vector of one (layer, sequence, KV head, path slot)
// row, for K and V together, all layers in one launch; consecutive threads
// move consecutive 16-byte pieces of the same row, so every warp reads and
// writes whole 256-byte rows.  Tree rows live in a separate scratch, so the
// gather never reads a row it also writes.
#include "gv_internal.cuh"

namespace gv {

__global__ void __launch_bounds__(256)
kv_compact_kernel(int L, int B, int N, int W, int Hkv, int S_max, int row_vec,
                  const uint4* __restrict__ treeK, const uint4* __restrict__ treeV,
                  uint4* __restrict__ cacheK, uint4* __restrict__ cacheV,
                  const int32_t* __restrict__ path, const int32_t* __restrict__ accept_len,
                  const int32_t* __restrict__ prefix_len, int32_t* __restrict__ new_len,
                  int32_t* __restrict__ seq_status) {
    pdl_wait();
    pdl_trigger();
    // Status / new_len: decided by block 0 from the same inputs every copying
    // thread tests, so the status write never changes another thread's choice.
    if (blockIdx.x == 0) {
        for (int b = threadIdx.x; b < B; b += blockDim.x) {
            const int P = prefix_len[b];
            const int n = accept_len[b];
            const int st = seq_status[b];
            if (st != GV_OK) {
                new_len[b] = P;
            } else if (P < 0 || n < 0 || P + n > S_max) {
                new_len[b] = P;
                seq_status[b] = GV_ERR_CAPACITY;
            } else {
                new_len[b] = P + n;
            }
        }
    }
    const size_t total = (size_t)L * B * Hkv * W * row_vec;
    for (size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (size_t)gridDim.x * blockDim.x) {
        const int v = (int)(idx % row_vec);
        size_t r = idx / row_vec;
        const int t = (int)(r % W);
        r /= W;
        const int h = (int)(r % Hkv);
        r /= Hkv;
        const int b = (int)(r % B);
        const int l = (int)(r / B);
        const int n = accept_len[b];
        if (t >= n) continue;
        const int P = prefix_len[b];
        if (P < 0 || P + n > S_max) continue;
        // Block 0 writes GV_ERR_CAPACITY only for sequences that fail the
        // test above, so reading the status before or after that write gives
        // the same decision here.
        if (seq_status[b] != GV_OK) continue;
        const int src = path[(size_t)b * W + t];
        if (src < 0 || src >= N) continue;
        const size_t lbh = ((size_t)l * B + b) * Hkv + h;
        const size_t dst = (lbh * S_max + (size_t)(P + t)) * row_vec + v;
        const size_t srcv = (lbh * N + (size_t)src) * row_vec + v;
        cacheK[dst] = treeK[srcv];
        cacheV[dst] = treeV[srcv];
    }
}

int launch_kv_compact(int L, int B, int N, int D, int Hkv, int d, int S_max, int esize,
                      const void* treeK, const void* treeV, void* cacheK, void* cacheV,
                      const int32_t* path, const int32_t* accept_len, const int32_t* prefix_len,
                      int32_t* new_len, int32_t* seq_status, cudaStream_t st) {
    const int W = D + 1;
    const int row_vec = d * esize / 16;
    const size_t total = (size_t)L * B * Hkv * W * row_vec;
    size_t blocks = (total + 255) / 256;
    const size_t cap = (size_t)sm_count() * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    launch_pdl(kv_compact_kernel, dim3((unsigned)blocks), dim3(256), 0, st, L, B, N, W, Hkv, S_max, row_vec,
               static_cast<const uint4*>(treeK), static_cast<const uint4*>(treeV),
               static_cast<uint4*>(cacheK), static_cast<uint4*>(cacheV), path, accept_len, prefix_len,
               new_len, seq_status);
    return check_launch("kv_compact_kernel");
}

}  // namespace gv
