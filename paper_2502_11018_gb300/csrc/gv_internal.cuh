// Internal helpers of libgv.so (not part of the C ABI).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "gv.h"

namespace gv {

// ---- host-side error bookkeeping -------------------------------------------
void set_error(const char* fmt, ...);
void clear_error();

#define GV_CHECK_ARG(cond, ...)                                     \
    do {                                                            \
        if (!(cond)) {                                              \
            ::gv::set_error(__VA_ARGS__);                           \
            return GV_ERR_ARG;                                      \
        }                                                           \
    } while (0)

// Launch-error check after a kernel launch.
int check_launch(const char* what);

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

inline cudaStream_t as_stream(void* s) { return reinterpret_cast<cudaStream_t>(s); }

// Number of SMs of the current device (cached per device).
int sm_count();
// Compute capability major*10+minor of the current device.
int device_cc();

// ---- programmatic dependent launch -------------------------------------------
// The step's kernels are launched with programmatic stream serialization, so a
// kernel's CTAs can be resident (and run their prologue) while the previous
// kernel of the stream finishes.  A kernel calls pdl_wait() before it reads
// anything an earlier kernel of the stream wrote, or writes anything one may
// still read: it returns once those grids have completed and their memory is
// visible.  pdl_trigger() lets the next kernel's CTAs launch; kernels that
// trigger only after their own pdl_wait() keep the ordering transitive (the
// next kernel starts after the previous one has completed).
//
// The split-K reduce kernels of the projections trigger before their wait, so
// that the next projection's CTAs can take the SMs the current GEMM frees and
// stream their first weight stages during its tail.  Their dependents (a
// projection, the tree attention, the LM head) read nothing before their own
// wait but constant weights and the KV cache of an earlier step; after it,
// the reduce has completed, and with it the GEMM it waited for.  A dependent
// grid launches only once every CTA of its primary has triggered, so no
// grid's CTAs can be kept off the SMs by a later grid's.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t st, Args... args) {
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// ---- device helpers ---------------------------------------------------------
constexpr unsigned FULL = 0xffffffffu;

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T> __device__ __forceinline__ T from_f32(float x);
template <> __device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) {
    return __float2bfloat16_rn(x);
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(FULL, v, o));
    return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FULL, v, o);
    return v;
}

// (value, id) ordering used by every selection: larger value first, then
// smaller id.  NaN never wins.
__device__ __forceinline__ bool better(float va, int ia, float vb, int ib) {
    return (va > vb) || (va == vb && ia < ib) || (vb != vb && va == va);
}

// One skinny projection out = epilogue(x W^T + bias) on the tensor cores
// (linear_sm103.cu).  The input may come in two column blocks: x holds
// columns [0, k_split) and x2 columns [k_split, K) (k_split % 64 == 0), so
// that a concatenation [a ; b] W^T is never materialised.
struct LinearOp {
    const void* x = nullptr;        // bf16 [rows][k_split], or [rows][K] when x2 is null
    const void* x2 = nullptr;       // bf16 [rows][K - k_split] or null
    int k_split = 0;
    const void* W = nullptr;        // bf16 [N][K], N = n_out (2 * n_out for SwiGLU)
    int rows = 0, K = 0, n_out = 0, epi = GV_LINEAR_STORE;
    const void* bias = nullptr;     // bf16 [N], added to the sums before the epilogue, or null
    const void* residual = nullptr; // bf16 [rows][n_out] (GV_LINEAR_ADD)
    void* out = nullptr;            // bf16 [rows][n0 or n_out]
    void* out1 = nullptr;           // column split of the stored output (n1 > 0)
    void* out2 = nullptr;
    int n0 = 0, n1 = 0;
    const void* norm_w = nullptr;   // fused RMSNorm of the ADD result (norm_out non-null)
    float eps = 0.f;
    void* norm_out = nullptr;
    void* ws = nullptr;             // fp32 partial sums, linear_workspace_bytes
};
size_t linear_workspace_bytes(int rows, int K, int N);
// The GEMM alone: writes the fp32 partial sums part[KS][rows][N] to op.ws and
// returns KS through *ks (the op's epilogue fields are ignored).
int launch_gemm_partials(const LinearOp& op, cudaStream_t st, int* ks);
int launch_linear(const LinearOp& op, cudaStream_t st);

// Per-(slot, row) partial results of the LM-head selection, merged by
// lmhead_merge_kernel.  Layout in the workspace (slots = producing tiles):
//   float val[slots][rows][K]; int id[slots][rows][K];  (top-K, K = k or 1)
//   float m[slots][rows]; float s[slots][rows];          (logits mode: max, sum exp)
struct SelectPartials {
    float* val;
    int* id;
    float* m;
    float* s;
    int slots;
    int rows;
    int K;
};

}  // namespace gv
