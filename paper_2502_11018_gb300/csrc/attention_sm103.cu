// gv_verify_attention, bf16 tensor-core path for sm_103a.
//
// GRIFFIN Section 3: every draft token is verified in one target forward
// pass; in each attention layer tree node i attends to the cached prefix and
// to the nodes on its own root chain (Section 4.1: rejecting a token drops
// its subtree, so the ancestor set is exactly what node i may see).
//
// Query rows: row r = i * G + hl of KV head g holds tree node i and query
// head g * G + hl; all G * N rows of (b, g) share every K/V block (GQA), and
// each 128 of them form one MMA M tile.  A unit = (sequence b, KV head g, M
// tile); each unit gets C CTAs (key splits).  The keys of (b, g) are cut into
// 128-key blocks: ceil(P_b / 128) prefix blocks and one tree block (the N <= 64
// tree keys, masked per query row by its ancestor bitmask).  The last split
// runs the tree block first and then the last prefix blocks; the others take
// the remaining prefix blocks round robin.
//
// Per block j of a CTA:
//   S_j = Q K_j^T          tcgen05.mma, Q and K K-major 128B-swizzled in smem,
//                          fp32 S in TMEM (three buffers: S_{j+1} and S_{j+2}
//                          can be computed during the softmax of block j)
//   softmax                two threads per query row, one per 64-key half of
//                          the block, read their S row half from TMEM, mask
//                          with a branch-free validity mask (prefix end, or
//                          the row's ancestor bitmask), exchange their half
//                          maxima through shared memory, keep the row's
//                          running max in the log2 domain and rescale O only
//                          when the max grew by more than 2^8 (exact: O and l
//                          always share one max), and write P = exp2(s - m) as
//                          bf16 back to TMEM, over the first half of its own S
//                          columns
//   O += P_j V_j           tcgen05.mma with A = P read from TMEM, V MN-major
//                          in smem (d contiguous), one accumulator per row tile
// Each CTA then writes o = O / l (bf16) and
// lse = m + log2(l) of its rows to the workspace (L2-resident), and
// attn_merge_kernel, launched right behind it, combines the C splits of every
// row into the bf16 output.  No CTA waits for another, so the splits need no
// cluster co-scheduling and the grid fills the SMs.
//
// Warp roles: warp 0 issues the TMA loads (lane 0 the K halves of the
// blocks and the raw Q tile, lane 1 the V halves); warp 1 owns TMEM and
// issues the MMAs; warps 2..9 rotate Q in place
// (RoPE from the per-step table), build the tree K/V tile, and run the
// softmax and the staging.
//
// Both kernels use programmatic dependent launch.  Before griddepcontrol.wait
// a CTA only initialises barriers and TMEM, reads step inputs written two
// launches before the step's first attention launch (ancestor masks, prefix
// lengths) and fills its K/V ring from the cache; the RoPE table, queries,
// tree keys/values, the workspace and the output are touched after it.  Every
// mbarrier wait is bounded; a CTA that gives up writes NaN lse for its rows,
// which turns the affected outputs into NaN.
#include "gv_internal.cuh"
#include "attention.cuh"
#include "attn_common.cuh"
#include "sm103.cuh"

namespace gv {
using namespace sm103;

constexpr int AT_BK = 128;                  // keys per block
constexpr int AT_HK = AT_BK / 2;            // keys per half (one softmax thread)
constexpr int AT_QHALF = 128 * 128;         // one M tile, 64 of the 128 d columns (bf16)
constexpr int AT_QTILE = 2 * AT_QHALF;      // one M tile of Q
constexpr int AT_KV_HALF = AT_BK * 128;     // 128 keys x 64 d bf16 (one swizzle sub-tile)
constexpr int AT_STAGE = 4 * AT_KV_HALF;    // K (2 halves) + V (2 halves)

// Softmax warps 2..9: warp w reads TMEM lane quarter (w & 3), i.e. query
// rows 32 * (w & 3) .. + 31, and key half h = (w - 2) >> 2 (keys 64h .. 64h+63)
// of every 128-key block, so each thread handles 64 scores per block.  The
// two threads of a row (warps w and w + 4) share the row's running max --
// they exchange their half maxima every block -- and one O accumulator; each
// keeps the sum of its own half, and the sums are added when the CTA's
// partial row is staged.
constexpr int AT_NSM = 256;               // softmax threads: 128 rows x 2 key halves
constexpr int AT_NTH = 64 + AT_NSM;       // + TMA producer warp + MMA warp
constexpr int AT_ST = 3;                  // K/V stages (64 KB each)
constexpr int AT_SB = 3;                  // S buffers in TMEM (128 columns each)
constexpr uint32_t AT_OCOL = 384;         // O at columns [384, 512)
constexpr uint32_t AT_TMEM_COLS = 512;    // S buffers [0, 384), O

// DIRECT: a single key split (C == 1) writes the final rows to the output
// itself (no partials, no merge kernel).
template <bool DIRECT>
__global__ void __launch_bounds__(AT_NTH, 1)
attn_tc_kernel(const __grid_constant__ CUtensorMap map_k, const __grid_constant__ CUtensorMap map_v,
               const __grid_constant__ CUtensorMap map_q, AttnArgs a) {
    constexpr int NSM = AT_NSM, ST = AT_ST;
    const int C = a.csize;                     // key splits per unit
    // CTA -> unit (sequence b, KV head g, M tile of 128 query rows) and key
    // split `rank` of that unit.
    const int cl = blockIdx.x / C;
    const int rank = blockIdx.x - cl * C;
    const int bg = cl / a.tiles;
    const int tile0 = cl % a.tiles;
    const int b = bg / a.Hkv, g = bg % a.Hkv;
    // prefix_len is a step input written before the previous kernel in the
    // stream started, so it may be read before griddepcontrol.wait.
    const int P = min(max(a.prefix_len[b], 0), a.S_max);
    const int nb_pre = (P + AT_BK - 1) / AT_BK;
    // The tree block goes to the last split and runs first there; it counts
    // as two blocks (its tile is built from the tree's keys and values on the
    // critical path).  The last split takes the last nt prefix blocks, the
    // other splits the first `rest` blocks round robin.
    const bool has_tree = rank == C - 1;
    const int per = (nb_pre + 2 + C - 1) / C;
    const int nt = C == 1 ? nb_pre : max(0, min(nb_pre, per - 2));
    const int rest = nb_pre - nt;
    const int nblk = has_tree ? nt + 1 : (rest > rank ? (rest - 1 - rank) / (C - 1) + 1 : 0);
    const int nb_per_tile = 128 / a.G;                   // nodes per M tile
    const int row0 = tile0 * 128;                        // first query row of this cluster
    const int R = min(a.G * a.N - row0, 128);            // query rows of this unit
    // Prefix block index of this CTA's j-th block (-1 for the tree block).
    auto prefix_block = [&](int j) -> int {
        if (has_tree) return j == 0 ? -1 : rest + (j - 1);
        return rank + (C - 1) * j;
    };

    // The 128B-swizzled tiles need 1024-byte alignment; the dynamic shared
    // memory of a kernel without static shared memory starts there (checked
    // below: a CTA whose base is not aligned gives up, with NaN rows).  No
    // slack is allocated, so that one merge CTA fits on the SM beside this one.
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = smem_raw;
    uint8_t* sQ = smem;                                  // 32 KB
    uint8_t* sKV = sQ + AT_QTILE;                        // ST x 64 KB
    // [2][128] (m, l) per key half, in the P area once the last PV is done
    float2* sML = reinterpret_cast<float2*>(sKV);    // [2][128] (m, l), once the ring is idle
    uint64_t* bars = reinterpret_cast<uint64_t*>(sKV + ST * AT_STAGE);
    // K and V of a stage land and are released separately: S_j frees K_j,
    // PV_j frees V_j, so the next K block can stream in during PV_j.
    uint64_t* k_full = bars;
    uint64_t* v_full = k_full + ST;
    uint64_t* k_empty = v_full + ST;
    uint64_t* v_empty = k_empty + ST;
    uint64_t* s_full = v_empty + ST;
    uint64_t* p_full = s_full + AT_SB;
    uint64_t* o_done = p_full + AT_SB;
    uint64_t* q_raw = o_done + AT_SB;
    uint64_t* q_full = q_raw + 1;
    uint64_t* drain = q_full + 1;
    uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
    // (cos, sin) of pairs 8c + 2q, 8c + 2q + 1 of node n of sequence b, read
    // from the per-step RoPE table (L2-resident: every CTA of the sequence
    // reads the same N x 512 B).
    // (no table: the queries and tree keys arrive rotated, gv_rope_apply)
    const bool rotate = a.rope != nullptr;
    const float4* rope_b = reinterpret_cast<const float4*>(a.rope) + (size_t)b * a.N * 32;
    auto rope_cs = [&](int n, int c, int q) -> float4 { return __ldg(rope_b + n * 32 + c * 4 + q); };
    volatile int* abort = reinterpret_cast<volatile int*>(tmem_holder + 1);
    // Half maxima of the current block, [block parity][key half][row], rounded
    // up to bf16 (both threads of a row then compute the same row max).
    __nv_bfloat16* sMX = reinterpret_cast<__nv_bfloat16*>(reinterpret_cast<uint8_t*>(tmem_holder) + 16);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < ST; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&v_full[s], 1);
            mbar_init(&k_empty[s], 1);
            mbar_init(&v_empty[s], 1);
        }
        for (int c = 0; c < AT_SB; ++c) {
            mbar_init(&s_full[c], 1);
            mbar_init(&p_full[c], NSM / 32);
            mbar_init(&o_done[c], 1);
        }
        mbar_init(q_raw, 1);
        mbar_init(q_full, 1);
        mbar_init(drain, 1);
        *abort = (smem_u32(smem_raw) & 1023u) != 0 ? 1 : 0;
        fence_mbar_init();
        if (nblk > 0) {
            prefetch_tmap(&map_q);
            prefetch_tmap(&map_k);
            prefetch_tmap(&map_v);
        }
    }
    if (warp == 1) tmem_alloc(tmem_holder, AT_TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_holder;
    pdl_trigger();

    // Row and key half of a softmax thread (valid for warps >= 2).
    const int t = threadIdx.x - 64;
    const int kh = warp >= 2 ? (warp - 2) >> 2 : 0;     // key half
    const int sub = warp & 3;                            // TMEM lane quarter
    const int row = sub * 32 + lane;                     // query row in the cluster's tile
    const int node = tile0 * nb_per_tile + row / a.G;    // tree node of this row
    const bool row_ok = warp >= 2 && node < a.N;
    const uint32_t lane_base = tmem + ((uint32_t)(sub * 32) << 16);
    const uint32_t ocol_self = lane_base + AT_OCOL + 64u * (uint32_t)kh;   // this thread's d columns of O
    float m_used = -INFINITY, l = 0.f;
    bool ok = true;

    if (nblk > 0) {
        if (warp == 0) {
            // ----------------------------------------------------- TMA producer
            // Lane 0 streams the K halves of the blocks (and the queries),
            // lane 1 the V halves, each as soon as its half of the stage is free.
            if (lane < 2) {
                const bool isk = lane == 0;
                uint64_t* full = isk ? k_full : v_full;
                uint64_t* empty = isk ? k_empty : v_empty;
                const CUtensorMap* map = isk ? &map_k : &map_v;
                const int off = isk ? 0 : 2 * AT_KV_HALF;
                const uint64_t pol_kv = policy_evict_first();
                const uint64_t pol_q = policy_evict_last();
                int issued[ST];
                for (int q = 0; q < ST; ++q) issued[q] = -1;
                bool q_issued = false;
                auto issue_q = [&]() {
                    pdl_wait();
                    // The box holds min(128 / G, N) nodes (the rows of nodes past
                    // it are never valid query rows).
                    mbar_arrive_expect_tx(q_raw, (uint32_t)(256 * a.G * min(nb_per_tile, a.N)));
                    const int z = b * a.N + tile0 * nb_per_tile;
                    tma_load_3d(sQ, &map_q, q_raw, 0, g * a.G, z, pol_q);
                    tma_load_3d(sQ + AT_QHALF, &map_q, q_raw, 64, g * a.G, z, pol_q);
                    q_issued = true;
                };
                for (int j = 0; j < nblk; ++j) {
                    const int s = j % ST;
                    const uint32_t ph = (uint32_t)(j / ST) & 1u;
                    // The first fill of the K/V ring streams before the
                    // dependency wait (the previous grid is still finishing),
                    // then the queries, then the remaining blocks.
                    if (isk && j == ST) issue_q();
                    const int k = prefix_block(j);
                    if (k < 0) continue;             // tree block: built by the softmax warps
                    if (!mbar_wait(&empty[s], ph ^ 1u, abort)) break;
                    mbar_arrive_expect_tx(&full[s], 2 * AT_KV_HALF);
                    uint8_t* st = sKV + s * AT_STAGE + off;
                    const int y = bg * a.S_max + k * AT_BK;
                    tma_load_2d(st, map, &full[s], 0, y, pol_kv);
                    tma_load_2d(st + AT_KV_HALF, map, &full[s], 64, y, pol_kv);
                    issued[s] = (int)ph;
                }
                if (isk && !q_issued && !*abort) issue_q();
                if (*abort) {
                    for (int q = 0; q < ST; ++q)
                        if (issued[q] >= 0) mbar_wait_timeout_only(&full[q], (uint32_t)issued[q]);
                    if (q_issued) mbar_wait_timeout_only(q_raw, 0);
                }
            }
        } else if (warp == 1) {
            // ------------------------------------------------------- MMA issuer
            if (lane == 0) {
                const uint32_t idesc_s = idesc_bf16(128, AT_BK);
                const uint32_t idesc_o = idesc_bf16(128, 128, /*b_mn_major=*/true);
                // (queries that arrive rotated are used as the copy lands them)
                bool mok = mbar_wait(rotate ? q_full : q_raw, 0, abort);
                tc_fence_after();
                // S_j = Q K_j^T into S buffer j % 3, as soon as block j's K
                // has landed and PV_{j-3} has consumed that buffer.
                auto issue_s = [&](int jj) {
                    const int s = jj % ST, buf = jj % AT_SB;
                    const uint32_t kbase = smem_u32(sKV + s * AT_STAGE);
#pragma unroll
                    for (int kb = 0; kb < 2; ++kb) {
                        const uint64_t qdesc = sdesc_kmajor_sw128(smem_u32(sQ + kb * AT_QHALF));
                        const uint64_t kdesc = sdesc_kmajor_sw128(kbase + kb * AT_KV_HALF);
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            mma_bf16(tmem + (uint32_t)(buf * AT_BK), qdesc + 2u * kk, kdesc + 2u * kk,
                                     idesc_s, (kb | kk) != 0);
                    }
                    mma_commit(&k_empty[s]);
                    mma_commit(&s_full[buf]);
                };
                // O += P_j V_j once softmax j has written P_j, with P read
                // from TMEM: the softmax stores the P of each key half (bf16
                // pairs, 16 columns) over the first half of that half's 64 S
                // columns.
                auto issue_pv = [&](int jj) {
                    const int pb = jj % AT_SB, sp = jj % ST, buf = jj % AT_SB;
                    // V as the MN-major B operand: rows = keys (128 B apart, SBO =
                    // 1 KB per 8 keys), the two 64-wide halves of d LBO = 8 KB apart.
                    uint64_t vdesc = sdesc_kmajor_sw128(smem_u32(sKV + sp * AT_STAGE + 2 * AT_KV_HALF));
                    vdesc = (vdesc & ~(0x3FFFull << 16)) | ((uint64_t)(AT_KV_HALF >> 4) << 16);
                    // One K step of 16 keys is 8 TMEM columns of P: keys 16 kk ..
                    // of half kk / 4 start at column 64 (kk / 4) + 8 (kk % 4).
#pragma unroll
                    for (int kk = 0; kk < AT_BK / 16; ++kk)
                        mma_bf16_ta(tmem + AT_OCOL, tmem + (uint32_t)(buf * AT_BK + AT_HK * (kk >> 2) + 8 * (kk & 3)),
                                    vdesc + (uint64_t)(kk * 128), idesc_o, (jj != 0) || (kk != 0));
                    mma_commit(&v_empty[sp]);
                    mma_commit(&o_done[pb]);
                };
                // Issue whichever is ready (S first: the softmax waits on it),
                // polling without blocking; give up after WAIT_TIMEOUT_NS
                // without progress.  S_j reuses the TMEM of S_{j-3} / P_{j-3}:
                // it is issued after PV_{j-3}, and the tensor pipe runs the
                // MMAs of this thread in order.
                int ns = 0, np = 0;
                unsigned long long t_last = globaltimer();
                while (mok && np < nblk) {
                    bool prog = false;
                    if (ns < nblk && np > ns - AT_SB &&
                        mbar_test_wait(&k_full[ns % ST], (uint32_t)(ns / ST) & 1u)) {
                        tc_fence_after();
                        issue_s(ns++);
                        prog = true;
                    }
                    if (np < ns && mbar_test_wait(&p_full[np % AT_SB], (uint32_t)(np / AT_SB) & 1u) &&
                        mbar_test_wait(&v_full[np % ST], (uint32_t)(np / ST) & 1u)) {
                        tc_fence_after();
                        issue_pv(np++);
                        prog = true;
                    }
                    if (prog) {
                        t_last = globaltimer();
                    } else if (*abort || globaltimer() - t_last > WAIT_TIMEOUT_NS) {
                        *abort = 1;
                        mok = false;
                    }
                }
                mma_commit(drain);
                mbar_wait_timeout_only(drain, 0);
            }
        } else {
            // -------------------------- Q rotation, tree tile, softmax, epilogue
            // The ancestor masks were written two launches before the step's
            // first attention launch, so they are read before
            // griddepcontrol.wait; the RoPE table, the queries and the tree
            // keys/values come after it.
            const unsigned long long anc_row =
                (has_tree && row_ok) ? __ldg(a.anc + (size_t)b * a.N + node) : 0ull;
            pdl_wait();
            // This row's RoPE pairs (chunks 4 kh .. 4 kh + 3), in flight while
            // the queries land.
            float4 rcs[16];
#pragma unroll
            for (int c = 0; c < 4; ++c)
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    rcs[4 * c + q] = (rotate && row_ok) ? rope_cs(node, 4 * kh + c, q) : make_float4(0.f, 0.f, 0.f, 0.f);
            if (has_tree) {
                // Rotated tree keys and the values into stage 0 (and into the
                // tree K/V scratch in global memory for gv_kv_compact).
                uint8_t* st = sKV;
                for (int e = t; e < AT_BK * 8; e += NSM) {
                    const int j = e >> 3, c = e & 7;
                    uint4 klo = make_uint4(0, 0, 0, 0), khi = klo, vlo = klo, vhi = klo;
                    if (j < a.N) {
                        // (every row tile's cluster builds the tile; the first writes the scratch)
                        const size_t src = (((size_t)b * a.N + j) * a.Hkv + g) * 16;
                        const uint4* kr = reinterpret_cast<const uint4*>(a.k_new) + src;
                        const uint4* vr = reinterpret_cast<const uint4*>(a.v_new) + src;
                        const uint4 k0 = __ldg(kr + c), k1 = __ldg(kr + 8 + c);
                        vlo = __ldg(vr + c);
                        vhi = __ldg(vr + 8 + c);
                        if (rotate) {
                            float4 cs[4];
#pragma unroll
                            for (int q = 0; q < 4; ++q) cs[q] = rope_cs(j, c, q);
                            rope8(k0, k1, cs, klo, khi);
                        } else {
                            klo = k0;
                            khi = k1;
                        }
                        uint4* tk = reinterpret_cast<uint4*>(a.treeK) + ((size_t)bg * a.N + j) * 16;
                        uint4* tv = reinterpret_cast<uint4*>(a.treeV) + ((size_t)bg * a.N + j) * 16;
                        if (tile0 == 0) {
                            tk[c] = klo;
                            tk[8 + c] = khi;
                            tv[c] = vlo;
                            tv[8 + c] = vhi;
                        }
                    }
                    *reinterpret_cast<uint4*>(st + sw128(j, c)) = klo;
                    *reinterpret_cast<uint4*>(st + AT_KV_HALF + sw128(j, c)) = khi;
                    *reinterpret_cast<uint4*>(st + 2 * AT_KV_HALF + sw128(j, c)) = vlo;
                    *reinterpret_cast<uint4*>(st + 3 * AT_KV_HALF + sw128(j, c)) = vhi;
                }
                named_bar_sync(1, NSM);
                if (t == 0) {
                    fence_proxy_async_smem();
                    mbar_arrive(&k_full[0]);
                    mbar_arrive(&v_full[0]);
                }
            }
            // RoPE of this thread's half of its Q row (16-byte chunks 4 kh ..
            // 4 kh + 3 of both d halves), in place once the raw tile has
            // landed: loads first, the rotation in registers, then the stores.
            {
                const int w = mbar_wait(q_raw, 0, abort) ? 1 : 0;   // every lane observes the copy
                if (__all_sync(FULL, w) && ok && rotate) {
                    uint4 lo[4], hi[4];
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        lo[c] = *reinterpret_cast<const uint4*>(sQ + sw128(row, 4 * kh + c));
                        hi[c] = *reinterpret_cast<const uint4*>(sQ + AT_QHALF + sw128(row, 4 * kh + c));
                    }
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        uint4 olo = make_uint4(0, 0, 0, 0), ohi = olo;
                        if (row_ok) rope8(lo[c], hi[c], &rcs[4 * c], olo, ohi);
                        lo[c] = olo;
                        hi[c] = ohi;
                    }
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        *reinterpret_cast<uint4*>(sQ + sw128(row, 4 * kh + c)) = lo[c];
                        *reinterpret_cast<uint4*>(sQ + AT_QHALF + sw128(row, 4 * kh + c)) = hi[c];
                    }
                }
                named_bar_sync(1, NSM);
                if (t == 0) {
                    fence_proxy_async_smem();
                    mbar_arrive(q_full);
                }
            }
            const float sl2 = a.scale * 1.4426950408889634f;     // scale * log2(e)
            for (int j = 0; j < nblk; ++j) {
                const int buf = j % AT_SB, s = j % ST;
                int w = ok ? 1 : 0;
                if (w && lane == 0) w = mbar_wait(&s_full[buf], (uint32_t)(j / AT_SB) & 1u, abort);
                w = __shfl_sync(FULL, w, 0);
                __syncwarp();
                tc_fence_after();
                uint32_t sv[AT_HK];
                tmem_ld32(lane_base + (uint32_t)(buf * AT_BK + AT_HK * kh), *reinterpret_cast<uint32_t(*)[32]>(&sv[0]));
                tmem_ld32(lane_base + (uint32_t)(buf * AT_BK + AT_HK * kh + 32),
                          *reinterpret_cast<uint32_t(*)[32]>(&sv[32]));
                tmem_wait_ld();
#pragma unroll
                for (int c = 0; c < AT_HK; ++c) asm volatile("" : "+r"(sv[c]));  // uses stay after the wait
                // Keys of the block this row may see: all of a full prefix block
                // (the common, unmasked path), else a branch-free mask (the
                // prefix end, or the row's ancestor bitmask); masked scores
                // become -inf and their exp2 is exactly 0.
                const int k = prefix_block(j);
                const int nvalid = k < 0 ? a.N : min(AT_BK, P - k * AT_BK);
                if (k < 0 || nvalid < AT_BK) {
                    // (the tree keys are nodes 0..N-1 <= 63: the first half)
                    unsigned long long vbits;
                    if (k < 0) {
                        vbits = kh == 0 ? anc_row : 0ull;
                    } else {
                        const int nv = nvalid - AT_HK * kh;  // valid keys of this half
                        vbits = nv >= 64 ? ~0ull : (nv <= 0 ? 0ull : ((1ull << nv) - 1ull));
                    }
                    const uint32_t vlo = (uint32_t)vbits, vhi = (uint32_t)(vbits >> 32);
#pragma unroll
                    for (int c = 0; c < AT_HK; ++c)
                        sv[c] = ((c < 32 ? vlo >> c : vhi >> (c - 32)) & 1u) ? sv[c] : __float_as_uint(-INFINITY);
                }
                float mxs[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
                for (int c = 0; c < AT_HK; c += 2)
                    mxs[(c >> 1) & 3] = max3(mxs[(c >> 1) & 3], __uint_as_float(sv[c]), __uint_as_float(sv[c + 1]));
                // This half's max, rounded up to bf16, to the row's other
                // thread (warp w +- 4, same lane) through shared memory; the
                // barrier of the pair also agrees on whether both got S_j.
                const __nv_bfloat16 mh =
                    __float2bfloat16_ru(max3(mxs[0], mxs[1], fmaxf(mxs[2], mxs[3])) * sl2);   // sl2 > 0
                __nv_bfloat16* mslot = sMX + (j & 1) * 256;
                mslot[kh * 128 + row] = mh;
                if (!pair_bar_and(2 + sub, w)) {
                    ok = false;
                    break;
                }
                const float mx = fmaxf(__bfloat162float(mh), __bfloat162float(mslot[(1 - kh) * 128 + row]));
                const float m_new = fmaxf(m_used, mx);
                const bool need = m_new > m_used + 8.0f;     // also true the first time
                float alpha = 1.0f;
                if (need) {
                    alpha = fast_exp2(m_used - m_new);       // 0 when m_used = -inf
                    m_used = m_new;
                }
                // p = 2^(s * sl2 - m); a row with no visible key so far keeps
                // m = -inf and all its p are 0 (the offset is then irrelevant).
                const float nmv = m_used == -INFINITY ? 0.f : -m_used;
                const uint64_t sc2 = f32x2(sl2, sl2), nm2 = f32x2(nmv, nmv);
                uint64_t ps[4] = {0ull, 0ull, 0ull, 0ull};
                uint32_t pk[AT_HK / 2];
#pragma unroll
                for (int c = 0; c < AT_HK / 2; ++c) {
                    const float2 xa = split_f32x2(ffma_f32x2(
                        f32x2(__uint_as_float(sv[2 * c]), __uint_as_float(sv[2 * c + 1])), sc2, nm2));
                    const float p0 = fast_exp2(xa.x), p1 = fast_exp2(xa.y);
                    ps[c & 3] = fadd_f32x2(ps[c & 3], f32x2(p0, p1));
                    pk[c] = pack_bf16(p0, p1);
                }
                const float2 psum = split_f32x2(fadd_f32x2(fadd_f32x2(ps[0], ps[1]), fadd_f32x2(ps[2], ps[3])));
                l = l * alpha + (psum.x + psum.y);
                const int pb = j % AT_SB;
                if (j >= 1 && __any_sync(FULL, need)) {
                    // Rescale this thread's 64 columns of O (the row's other
                    // thread takes the other 64, with the same alpha): PV_{j-1}
                    // must have landed first.  A failed wait is seen by both
                    // threads of the row at the next block's pair barrier.
                    if (lane == 0)
                        w = mbar_wait(&o_done[(j - 1) % AT_SB], (uint32_t)((j - 1) / AT_SB) & 1u, abort);
                    if (__shfl_sync(FULL, w, 0)) {
                        __syncwarp();
                        tc_fence_after();
#pragma unroll
                        for (int c0 = 0; c0 < 64; c0 += 32) {
                            uint32_t ov[32];
                            tmem_ld32(ocol_self + c0, ov);
                            tmem_wait_ld();
                            uint32_t lo[16], hi[16];
#pragma unroll
                            for (int e = 0; e < 16; ++e) {
                                lo[e] = __float_as_uint(__uint_as_float(ov[e]) * alpha);
                                hi[e] = __float_as_uint(__uint_as_float(ov[16 + e]) * alpha);
                            }
                            tmem_st16(ocol_self + c0, lo);
                            tmem_st16(ocol_self + c0 + 16, hi);
                        }
                        tmem_wait_st();
                    } else {
                        ok = false;
                    }
                }
                // P over the first 32 of this half's 64 S columns.
                tmem_st16(lane_base + (uint32_t)(buf * AT_BK + AT_HK * kh), *reinterpret_cast<uint32_t(*)[16]>(&pk[0]));
                tmem_st16(lane_base + (uint32_t)(buf * AT_BK + AT_HK * kh + 16),
                          *reinterpret_cast<uint32_t(*)[16]>(&pk[16]));
                const bool zero_v = k >= 0 && nvalid < AT_BK;
                if (zero_v && kh == 0) {
                    // Zero the V rows past the prefix end (they may hold anything).
                    int w2 = 1;
                    if (lane == 0) w2 = mbar_wait(&v_full[s], (uint32_t)(j / ST) & 1u, abort);
                    if (__shfl_sync(FULL, w2, 0)) {
                        uint8_t* vt = sKV + s * AT_STAGE + 2 * AT_KV_HALF;
                        for (int e = row; e < (AT_BK - nvalid) * 16; e += 128) {
                            const int key = nvalid + (e >> 4), c = e & 15;
                            *reinterpret_cast<uint4*>(vt + (c >> 3) * AT_KV_HALF + sw128(key, c & 7)) =
                                make_uint4(0, 0, 0, 0);
                        }
                    }
                }
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    if (zero_v) fence_proxy_async_smem();   // the zeroed V rows, for the MMA
                    mbar_arrive(&p_full[pb]);
                }
            }
        }
    }

    // ------------------------------------------------ partial rows to the workspace
    // The row's normalised partial o = O / l, l the sum of both key halves'
    // sums (bf16, the 16-byte chunks of row r rotated by r & 15
    // so that the lanes of a warp store distinct banks) and lse = m + log2(l)
    // are staged in the (now free) Q and P areas, then written to the
    // workspace with one bulk copy each; attn_merge_kernel combines the C
    // splits of every row.  lse is -inf for a CTA without blocks and NaN for
    // one that gave up.
    uint8_t* stg = sQ;                                  // R rows x 256 B
    float* stg_lse = reinterpret_cast<float*>(sKV + 4096);   // R floats, once the ring is idle
    int w = 0;
    if (warp >= 2) {
        w = ok && nblk > 0 ? 1 : 0;
        if (w && lane == 0)
            w = mbar_wait(&o_done[(nblk - 1) % AT_SB], (uint32_t)((nblk - 1) / AT_SB) & 1u, abort);
        w = __shfl_sync(FULL, w, 0);
        sML[kh * 128 + row] = make_float2(m_used, l);
    }
    // The halves' (m, l) and the last PV are visible after this barrier; the
    // CTA's partial is valid only if every softmax warp finished.
    w = __syncthreads_and(warp < 2 || w);
    // The workspace may still be read by the previous grid (the merge of the
    // previous call): wait for it before writing (a no-op if already done).
    pdl_wait();
    if (warp >= 2) {
        const bool mine = row < R;
        const float2 other = sML[(1 - kh) * 128 + row];
        const float M = m_used;                 // the row's max, shared by its halves
        const float ltot = l + other.y;
        uint8_t* srow = stg + row * 256;
        // With a single key split the row is final: it goes straight to the
        // output ([B][N][Hq][d], bf16) and no merge kernel runs.
        uint4* orow = nullptr;
        if (DIRECT && mine) {
            const int r = row0 + row, i = r / a.G, h = g * a.G + r % a.G;
            orow = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(a.out) +
                                            (((size_t)b * a.N + i) * a.Hq + h) * 128);
        }
        if (w) {
            // This thread writes d columns [64 kh, 64 kh + 64) of the row.
            tc_fence_after();
            const float inv = ltot > 0.f ? 1.0f / ltot : 0.f;
#pragma unroll
            for (int c0 = 0; c0 < 64; c0 += 32) {
                uint32_t os[32];
                tmem_ld32(ocol_self + (uint32_t)c0, os);
                tmem_wait_ld();
                if (mine) {
#pragma unroll
                    for (int e = 0; e < 32; e += 8) {
                        const int ch = (64 * kh + c0 + e) >> 3;   // 16-byte chunk of the 256-byte row
                        float v[8];
#pragma unroll
                        for (int u = 0; u < 8; ++u) v[u] = __uint_as_float(os[e + u]) * inv;
                        const uint4 pv = make_uint4(pack_bf16(v[0], v[1]), pack_bf16(v[2], v[3]),
                                                    pack_bf16(v[4], v[5]), pack_bf16(v[6], v[7]));
                        if (DIRECT)
                            orow[ch] = pv;
                        else
                            *reinterpret_cast<uint4*>(srow + ((ch ^ (row & 15)) << 4)) = pv;
                    }
                }
            }
        }
        if (DIRECT && mine && !w) {
            // (the single split owns the tree block, so it gave up)
            const uint32_t nan2 = pack_bf16(NAN, NAN);
#pragma unroll
            for (int ch = 0; ch < 8; ++ch) orow[8 * kh + ch] = make_uint4(nan2, nan2, nan2, nan2);
        }
        if (mine && !DIRECT) {
            if (kh == 0)
                stg_lse[row] = w ? (ltot > 0.f ? M + log2f(ltot) : -INFINITY) : (nblk > 0 ? NAN : -INFINITY);
            if (!w) {
                // No partial (no blocks, or gave up): zeros, so that the
                // merge may weight every split without testing its weight.
#pragma unroll
                for (int ch = 0; ch < 8; ++ch)
                    *reinterpret_cast<uint4*>(srow + ((8 * kh + ch) << 4)) = make_uint4(0, 0, 0, 0);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (*abort) {
        // A role gave up, so a copy may have landed in the staging area after
        // the rows were staged (each role drains its own copies before the
        // barrier above): mark every row of this CTA invalid again.
        if (warp >= 2 && kh == 0 && row < R && !DIRECT) stg_lse[row] = NAN;
        if (warp >= 2 && row < R && DIRECT) {
            const int r = row0 + row, i = r / a.G, h = g * a.G + r % a.G;
            uint4* orow = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(a.out) +
                                                   (((size_t)b * a.N + i) * a.Hq + h) * 128);
            const uint32_t nan2 = pack_bf16(NAN, NAN);
            for (int ch = 0; ch < 8; ++ch) orow[8 * kh + ch] = make_uint4(nan2, nan2, nan2, nan2);
        }
        __syncthreads();
    }
    if (warp == 1) tmem_dealloc(tmem, AT_TMEM_COLS);
    if (threadIdx.x == 0 && !DIRECT) {
        fence_proxy_async_smem();   // the staged rows, for the bulk copies
        const size_t split = (size_t)cl * C + rank;
        bulk_store(static_cast<uint8_t*>(a.part_o_bf16) + split * 128 * 256, stg, (uint32_t)R * 256u);
        bulk_store(a.part_ml + split * 128, stg_lse, (uint32_t)((R + 3) & ~3) * 4u);
        bulk_commit();
        bulk_wait_read();           // the staging smem may be released; the writes
                                    // are visible to the grids that depend on this one
    }
}

// Combines the C key splits of every query row: one thread per (row, 16-byte
// chunk of d), weights 2^(lse_s - max lse) over the splits, bf16 output.
// Launched right after attn_tc_kernel with programmatic dependent launch; it
// reads the partials after griddepcontrol.wait.
constexpr int AM_ROWS = 16;                 // rows per CTA (x 16 chunks = 256 threads)

__global__ void __launch_bounds__(AM_ROWS * 16)
attn_merge_kernel(AttnArgs a) {
    pdl_trigger();
    const int C = a.csize;
    // ceil(min(128, G N) / AM_ROWS) CTAs per unit: one merge CTA per SM fits
    // beside an attention CTA, so a grid of at most one CTA per SM is resident
    // (and waiting) before the attention grid ends.
    const int per_unit = (min(128, a.G * a.N) + AM_ROWS - 1) / AM_ROWS;
    const int cl = blockIdx.x / per_unit;                // unit
    const int row = (blockIdx.x % per_unit) * AM_ROWS + (threadIdx.x >> 4);
    const int ch = threadIdx.x & 15;
    const int bg = cl / a.tiles, tile0 = cl % a.tiles;
    const int b = bg / a.Hkv, g = bg % a.Hkv;
    const int r = tile0 * 128 + row;                    // query row of (b, g)
    if (row >= 128 || r >= a.G * a.N) return;
    pdl_wait();
    const size_t split0 = (size_t)cl * C;
    // All loads first (the lse of every split, then its 16-byte chunk).
    float lsv[16];
    float M = -INFINITY;
    bool bad = false;
#pragma unroll
    for (int q = 0; q < 16; ++q) {
        lsv[q] = q < C ? __ldcg(a.part_ml + (split0 + q) * 128 + row) : -INFINITY;
        bad |= lsv[q] != lsv[q];
        M = fmaxf(M, lsv[q]);
    }
    const uint8_t* po = static_cast<const uint8_t*>(a.part_o_bf16);
    const size_t off = (size_t)row * 256 + ((ch ^ (row & 15)) << 4);
    uint4 v[16];
#pragma unroll
    for (int q = 0; q < 16; ++q)
        if (q < C) v[q] = __ldcg(reinterpret_cast<const uint4*>(po + (split0 + q) * 128 * 256 + off));
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    float wsum = 0.f;
#pragma unroll
    for (int q = 0; q < 16; ++q) {
        if (q < C) {
            const float wq = lsv[q] == -INFINITY ? 0.f : fast_exp2(lsv[q] - M);
            wsum += wq;
            const uint32_t u[4] = {v[q].x, v[q].y, v[q].z, v[q].w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float2 f = unpack_bf16(u[e]);
                acc[2 * e] = fmaf(wq, f.x, acc[2 * e]);
                acc[2 * e + 1] = fmaf(wq, f.y, acc[2 * e + 1]);
            }
        }
    }
    const float inv = bad ? NAN : 1.0f / wsum;
    const int i = r / a.G, h = g * a.G + r % a.G;
    __nv_bfloat16* o = static_cast<__nv_bfloat16*>(a.out) + (((size_t)b * a.N + i) * a.Hq + h) * 128;
    reinterpret_cast<uint4*>(o)[ch] =
        make_uint4(pack_bf16(acc[0] * inv, acc[1] * inv), pack_bf16(acc[2] * inv, acc[3] * inv),
                   pack_bf16(acc[4] * inv, acc[5] * inv), pack_bf16(acc[6] * inv, acc[7] * inv));
}

// gv_rope_apply: the rotation the split kernel applies to its queries and tree
// keys (rope8, the same arithmetic), ahead of time for L layers.  One thread
// per (row, 16-byte chunk of the low half): rows are [L][B][N][H] of d = 128.
__global__ void __launch_bounds__(256)
rope_apply_kernel(const __nv_bfloat16* __restrict__ x, size_t layer_stride, int L, int B, int N, int H,
                  const float* __restrict__ rope, __nv_bfloat16* __restrict__ out) {
    pdl_wait();
    pdl_trigger();
    const size_t t = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    const size_t rows = (size_t)L * B * N * H;
    if (t >= rows * 8) return;
    const size_t row = t >> 3;
    const int c = (int)(t & 7);
    const int l = (int)(row / ((size_t)B * N * H));
    const size_t r = row - (size_t)l * B * N * H;          // (b, n, h) within the layer
    const size_t bn = r / H;                               // b * N + n
    const uint4* src = reinterpret_cast<const uint4*>(x + (size_t)l * layer_stride + r * 128);
    const uint4 lo = __ldg(src + c), hi = __ldg(src + 8 + c);
    const float4* cs = reinterpret_cast<const float4*>(rope) + bn * 32 + c * 4;
    float4 c4[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) c4[q] = __ldg(cs + q);
    uint4 olo, ohi;
    rope8(lo, hi, c4, olo, ohi);
    uint4* dst = reinterpret_cast<uint4*>(out) + row * 16;
    dst[c] = olo;
    dst[8 + c] = ohi;
}

int launch_rope_apply(const void* x, size_t layer_stride, int L, int B, int N, int H, const float* rope, void* out,
                      cudaStream_t st) {
    const size_t threads = (size_t)L * B * N * H * 8;
    if (threads == 0) return GV_OK;
    launch_pdl(rope_apply_kernel, dim3((unsigned)((threads + 255) / 256)), dim3(256), 0, st,
               static_cast<const __nv_bfloat16*>(x), layer_stride, L, B, N, H, rope, static_cast<__nv_bfloat16*>(out));
    return check_launch("rope_apply_kernel");
}

// ----------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn tensor_map_encoder();
int make_map_2d(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows,
                uint64_t row_stride_bytes);

// 3-D map over q[B*N][Hq][128] (bf16) with box {64 d, G heads, min(128/G, N)
// nodes}: the box lands in smem as up to 128 rows (node-major, head-minor) of
// 64 d.
static int make_map_q(CUtensorMap* map, const void* q, int BN, int Hq, int G, int N) {
    EncodeTiledFn enc = tensor_map_encoder();
    if (!enc) {
        set_error("cuTensorMapEncodeTiled unavailable");
        return GV_ERR_CUDA;
    }
    cuuint64_t dims[3] = {128, (cuuint64_t)Hq, (cuuint64_t)BN};
    cuuint64_t strides[2] = {256, (cuuint64_t)Hq * 256};
    cuuint32_t box[3] = {64, (cuuint32_t)G, (cuuint32_t)(128 / G < N ? 128 / G : N)};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(q), dims, strides,
                     box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        set_error("cuTensorMapEncodeTiled (q) failed (%d)", (int)r);
        return GV_ERR_CUDA;
    }
    return GV_OK;
}

static size_t attn_tc_smem() {
    return (size_t)AT_QTILE + (size_t)AT_ST * AT_STAGE + 8 * (4 * AT_ST + 3 * AT_SB + 3) + 16 +
           2 * 2 * 128 * sizeof(__nv_bfloat16);
}

// Key splits per unit (CTAs per (sequence, KV head, M tile)): as many as fit
// the SMs in one wave of 1-CTA-per-SM CTAs, at most 16, and at least 4 for
// long caches so that a long sequence of a ragged batch is not one CTA's
// serial work; never more than the blocks a unit can have.  The workspace
// plan uses the same count.
int attn_tc_splits(int units, int S_max) {
    int c = sm_count() / units;
    if (S_max >= 4096 && c < 4) c = 4;
    const int blocks = (S_max + AT_BK - 1) / AT_BK + 1;   // most blocks a unit can have
    if (c > blocks) c = blocks;
    if (c > 16) c = 16;
    if (c < 1) c = 1;
    return c;
}

int launch_attn_tc(const AttnArgs& a0, cudaStream_t st, int phase) {
    const int units = a0.B * a0.Hkv * a0.tiles;
    if (!(phase & 1)) {
        if (a0.csize == 1) return GV_OK;   // the split kernel wrote the output
        const int rmax = a0.G * a0.N < 128 ? a0.G * a0.N : 128;
        cudaError_t e = launch_pdl(attn_merge_kernel, dim3((unsigned)(units * ((rmax + AM_ROWS - 1) / AM_ROWS))),
                                   dim3(AM_ROWS * 16), 0, st, a0);
        if (e != cudaSuccess) {
            set_error("attn_merge_kernel launch: %s", cudaGetErrorString(e));
            return GV_ERR_CUDA;
        }
        return GV_OK;
    }
    CUtensorMap mk, mv, mq;
    const uint64_t rows = (uint64_t)a0.B * a0.Hkv * a0.S_max;
    int rc = make_map_2d(&mk, a0.cacheK, rows, 128, AT_BK, 256);
    if (rc != GV_OK) return rc;
    rc = make_map_2d(&mv, a0.cacheV, rows, 128, AT_BK, 256);
    if (rc != GV_OK) return rc;
    rc = make_map_q(&mq, a0.q, a0.B * a0.N, a0.Hq, a0.G, a0.N);
    if (rc != GV_OK) return rc;
    const size_t smem = attn_tc_smem();
    cudaFuncSetAttribute(attn_tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    cudaFuncSetAttribute(attn_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    cudaError_t e = a0.csize == 1
                        ? launch_pdl(attn_tc_kernel<true>, dim3((unsigned)units), dim3(AT_NTH), smem, st, mk, mv,
                                     mq, a0)
                        : launch_pdl(attn_tc_kernel<false>, dim3((unsigned)(units * a0.csize)), dim3(AT_NTH), smem,
                                     st, mk, mv, mq, a0);
    if (e != cudaSuccess) {
        set_error("attn_tc_kernel launch: %s", cudaGetErrorString(e));
        return GV_ERR_CUDA;
    }
    if (a0.csize == 1 || !(phase & 2)) return GV_OK;   // (one split: the split kernel wrote the output)
    const int rmax = a0.G * a0.N < 128 ? a0.G * a0.N : 128;
    e = launch_pdl(attn_merge_kernel, dim3((unsigned)(units * ((rmax + AM_ROWS - 1) / AM_ROWS))),
                   dim3(AM_ROWS * 16), 0, st, a0);
    if (e != cudaSuccess) {
        set_error("attn_merge_kernel launch: %s", cudaGetErrorString(e));
        return GV_ERR_CUDA;
    }
    return GV_OK;
}

}  // namespace gv
