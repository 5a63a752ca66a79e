// gv_tree_build: depths, RoPE positions and 64-bit ancestor masks of draft
// trees (GRIFFIN Appendix C dynamic tree; Section 4.1 subtree rejection).
//
// One 64-thread block per sequence, thread i = node i.  The ancestor set is
// built by pointer jumping: thread i holds the set of nodes from i up to (not
// including) its current jump target, and each round unions in the jump
// target's set and doubles the jump, so six rounds cover any depth <= 63.
#include "gv_internal.cuh"

namespace gv {

__global__ void __launch_bounds__(64)
tree_build_kernel(const int32_t* __restrict__ parents, const int32_t* __restrict__ prefix_len,
                  int N, int32_t* __restrict__ depth, int32_t* __restrict__ pos,
                  unsigned long long* __restrict__ anc, int32_t* __restrict__ seq_status) {
    __shared__ int s_jump[64];
    __shared__ unsigned long long s_set[64];
    pdl_wait();
    pdl_trigger();
    const int b = blockIdx.x;
    const int i = threadIdx.x;
    int jump = -1;
    bool bad = false;
    if (i < N) {
        jump = parents[(size_t)b * N + i];
        bad = (i == 0) ? (jump != -1) : (jump < 0 || jump >= i);
    }
    const int any_bad = __syncthreads_or(bad);
    const int P = prefix_len[b];
    unsigned long long set = (i < N) ? (1ull << i) : 0ull;
    if (!any_bad) {
#pragma unroll 1
        for (int round = 0; round < 6; ++round) {
            if (i < N) {
                s_jump[i] = jump;
                s_set[i] = set;
            }
            __syncthreads();
            if (i < N && jump >= 0) {
                set |= s_set[jump];
                jump = s_jump[jump];
            }
            __syncthreads();
        }
    }
    if (i < N) {
        const size_t o = (size_t)b * N + i;
        const int dep = any_bad ? 0 : (__popcll(set) - 1);
        depth[o] = dep;
        pos[o] = P + dep;
        anc[o] = set;
        if (i == 0) seq_status[b] = any_bad ? GV_ERR_INVALID_TREE : GV_OK;
    }
}

int launch_tree_build(const int32_t* parents, const int32_t* prefix_len, int B, int N,
                      int32_t* depth, int32_t* pos, uint64_t* anc, int32_t* seq_status,
                      cudaStream_t st) {
    launch_pdl(tree_build_kernel, dim3(B), dim3(64), 0, st, parents, prefix_len, N, depth, pos,
               reinterpret_cast<unsigned long long*>(anc), seq_status);
    return check_launch("tree_build_kernel");
}

}  // namespace gv
