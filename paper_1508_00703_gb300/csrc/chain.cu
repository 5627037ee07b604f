// Chain engine: pdb_sgd_epoch under a CHAIN schedule.
//
// When the conflict graph is close to one chain (a feature present in most
// examples makes every example depend on the one before), the concurrency
// the read and write constraints allow (Theorem 2) is about one example at a
// time, and what bounds the run is the latency of one dependency hop.  Here
// one thread block runs the examples strictly in data order -- the
// sequential computation of Algorithm 1 itself -- so a hop costs a few
// hundred cycles instead of a round trip through L2:
//
//   warp 0       computes example r (same fp32 operation order as the other
//                engines: lane i mod 32 accumulates element i with fused
//                multiply-adds, then the xor-shuffle combine), and pushes
//                each new weight whose next occurrence lies in one of the
//                next D examples straight into that example's weight slot;
//   warps 1-3,5-7 prefetch with cp.async (row bounds 7 steps ahead; ids,
//                values, labels and link words 4 steps ahead; the weights
//                nobody will push 2 steps ahead) and write the new weights of
//                the previous step through to global memory.
//
// A pipeline step handles G = 4 consecutive examples, so the fixed cost of a
// step (barrier, copy bookkeeping) is shared by four hops.
//
// Ordering: a pushed weight (next occurrence within D = 16 examples) is
// written by warp 0 before it computes the consumer (program order); a
// gathered weight's last writer lies more than D examples back, so its
// global store was issued at least one step before the gather, with
// __syncthreads between.  The pipeline drains at every epoch boundary.  No
// spin waits.
#include <cuda_runtime.h>

#include "common.cuh"

using namespace pdb;

namespace {

constexpr int CH_G = 4;                     // examples per pipeline step
constexpr int CH_DS = 4;                    // steps between ids/values prefetch and compute
constexpr int CH_BS = 2;                    // steps between weight gathers and compute
constexpr int CH_L = CH_DS + CH_BS + 1;     // steps between a row_ptr copy and its first use
constexpr int CH_D = CH_G * CH_DS;          // forwarding window (examples)
constexpr int CH_SLOTS = 32;                // example slots (power of two, > (CH_DS + 2) * CH_G)
constexpr int CH_MAXK = 256;                // longest example this engine takes
constexpr int CH_RP = 64;                   // row_ptr ring (power of two, > (CH_L + 2) * CH_G + 1)
constexpr int CH_THREADS = 256;
// Warps are spread over the SM's four schedulers by warp index mod 4, so
// warp 4 would compete with the computing warp 0 for issue slots: it only
// joins the barriers.  Warps 1-3 and 5-7 prefetch.
constexpr int CH_PF = CH_THREADS - 64;      // prefetching threads
constexpr int CH_PER = (CH_G * CH_MAXK + CH_PF - 1) / CH_PF;   // positions per prefetching thread per step
// link word of a position: bit 31 = its weight will be pushed by an earlier
// example (skip the gather); bit 30 = push the new weight to the next
// occurrence, which is element (bits 0..15) of the example (bits 16..23)
// examples later
constexpr uint32_t LK_RECV = 1u << 31, LK_PUSH = 1u << 30;
static_assert((CH_SLOTS & (CH_SLOTS - 1)) == 0 && (CH_RP & (CH_RP - 1)) == 0, "ring sizes must be powers of two");
static_assert(CH_SLOTS > (CH_DS + 2) * CH_G && CH_RP > (CH_L + 2) * CH_G + 1, "rings too short");
static_assert(CH_D < 256 && CH_MAXK <= 65536, "link word fields");
static_assert((CH_G & (CH_G - 1)) == 0, "examples per step must be a power of two");

struct ChainSmem {
    int32_t col[CH_SLOTS][CH_MAXK];
    float val[CH_SLOTS][CH_MAXK];
    uint32_t link[CH_SLOTS][CH_MAXK];
    float wp[CH_SLOTS][CH_MAXK];    // weight each element reads (gathered or pushed)
    float out[CH_SLOTS][CH_MAXK];   // weight each element writes
    int64_t rp[CH_RP];
    float y[CH_SLOTS];
};

__device__ __forceinline__ void cp4(void *smem_dst, const void *gsrc)
{
    const unsigned d = (unsigned)__cvta_generic_to_shared(smem_dst);
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(d), "l"(gsrc) : "memory");
}
__device__ __forceinline__ void cp8(void *smem_dst, const void *gsrc)
{
    const unsigned d = (unsigned)__cvta_generic_to_shared(smem_dst);
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(d), "l"(gsrc) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_wait_b() { asm volatile("cp.async.wait_group %0;" ::"n"(CH_BS - 1) : "memory"); }
__device__ __forceinline__ void cp_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// The positions of the CH_G examples of step t are contiguous: [rp[t*G], rp[t*G+G]).
// Element e of that range belongs to example r (found among the G bounds) at index i.
struct StepRange {
    int64_t b0;
    int total;
    int64_t bound[CH_G + 1];
};

__device__ __forceinline__ bool step_range(const ChainSmem &S, int t, int N, StepRange &R)
{
    const int r0 = t * CH_G;
    if (t < 0 || r0 >= N) return false;
#pragma unroll
    for (int j = 0; j <= CH_G; ++j) R.bound[j] = S.rp[min(r0 + j, N) & (CH_RP - 1)];
    R.b0 = R.bound[0];
    R.total = (int)(R.bound[CH_G] - R.b0);
    return true;
}

__device__ __forceinline__ void locate(const StepRange &R, int t, int e, int &row, int &i)
{
    const int64_t pos = R.b0 + e;
    int j = 0;
#pragma unroll
    for (int q = 1; q < CH_G; ++q) j += pos >= R.bound[q];
    row = t * CH_G + j;
    i = (int)(pos - R.bound[j]);
}

template <int R>
__global__ __launch_bounds__(CH_THREADS, 1) void k_sgd_chain(int32_t n_rows, const int64_t *__restrict__ row_ptr,
                                                             const int32_t *__restrict__ col,
                                                             const float *__restrict__ val,
                                                             const float *__restrict__ y,
                                                             const uint32_t *__restrict__ link, float *w, int loss,
                                                             float eta, int epochs, int *status)
{
    extern __shared__ __align__(16) unsigned char smem_raw[];
    ChainSmem &S = *reinterpret_cast<ChainSmem *>(smem_raw);
    if (read_status(status)) return;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const bool compute = warp == 0, idle = warp == 4;
    const int ptid = tid - (warp < 4 ? 32 : 64);
    const int N = n_rows;
    const int steps = (N + CH_G - 1) / CH_G;

    for (int ep = 0; ep < epochs; ++ep) {
        for (int t = -CH_L; t <= steps; ++t) {
            if (!compute && !idle) {
                StepRange R;
                // stage W: new weights of step t - 1 through to global memory; a weight that a
                // later example of the same step writes again is left to that example (two
                // stores of one step to one address would race)
                if (step_range(S, t - 1, N, R)) {
#pragma unroll
                    for (int u = 0; u < CH_PER; ++u) {
                        const int e = ptid + u * CH_PF;
                        if (e < R.total) {
                            int row, i;
                            locate(R, t - 1, e, row, i);
                            const int slot = row & (CH_SLOTS - 1);
                            const uint32_t l = S.link[slot][i];
                            const bool rewritten = (l & LK_PUSH) && (row & (CH_G - 1)) + (int)((l >> 16) & 0xffu) < CH_G;
                            if (!rewritten) w[S.col[slot][i]] = S.out[slot][i];
                        }
                    }
                }
                // stage R: row_ptr entries [(t+L)G, (t+L)G + G) with L = DS + BS + 1, so that
                // stage A of step t finds the bounds of step t + DS (and the entry after it) complete
                {
                    const int r = (t + CH_L) * CH_G + ptid;
                    if (ptid < CH_G && r >= 0 && r <= N) cp8(&S.rp[r & (CH_RP - 1)], row_ptr + r);
                }
                // stage A: ids, values, link words and labels of step t + DS
                if (step_range(S, t + CH_DS, N, R)) {
#pragma unroll
                    for (int u = 0; u < CH_PER; ++u) {
                        const int e = ptid + u * CH_PF;
                        if (e < R.total) {
                            int row, i;
                            locate(R, t + CH_DS, e, row, i);
                            const int slot = row & (CH_SLOTS - 1);
                            const int64_t pos = R.b0 + e;
                            cp4(&S.col[slot][i], col + pos);
                            cp4(&S.link[slot][i], link + pos);
                            if (val) cp4(&S.val[slot][i], val + pos);
                        }
                    }
                    const int r = (t + CH_DS) * CH_G + ptid;
                    if (ptid < CH_G && r < N) cp4(&S.y[r & (CH_SLOTS - 1)], y + r);
                }
                // stage B: weights of step t + BS that no recent example will push (the
                // thread that copied a position in stage A handles it here)
                if (step_range(S, t + CH_BS, N, R)) {
                    uint32_t l[CH_PER];
                    int32_t j[CH_PER];
                    int sl[CH_PER], ix[CH_PER];
#pragma unroll
                    for (int u = 0; u < CH_PER; ++u) {
                        const int e = ptid + u * CH_PF;
                        l[u] = LK_RECV;
                        j[u] = 0;
                        sl[u] = 0;
                        ix[u] = 0;
                        if (e < R.total) {
                            int row, i;
                            locate(R, t + CH_BS, e, row, i);
                            sl[u] = row & (CH_SLOTS - 1);
                            ix[u] = i;
                            l[u] = S.link[sl[u]][i];
                            j[u] = S.col[sl[u]][i];
                        }
                    }
#pragma unroll
                    for (int u = 0; u < CH_PER; ++u)
                        if (!(l[u] & LK_RECV)) cp4(&S.wp[sl[u]][ix[u]], w + j[u]);
                }
                cp_commit();
                cp_wait_b();
            } else if (t >= 0 && t < steps) {
                // compute the G examples of step t in data order
                for (int r = t * CH_G; r < min(N, t * CH_G + CH_G); ++r) {
                    const int slot = r & (CH_SLOTS - 1);
                    const int k = (int)(S.rp[(r + 1) & (CH_RP - 1)] - S.rp[r & (CH_RP - 1)]);
                    float xv[R], wv[R];
                    uint32_t lk[R];
                    float acc = 0.0f;
#pragma unroll
                    for (int q = 0; q < R; ++q) {
                        const int i = q * 32 + lane;
                        if (i < k) {
                            xv[q] = val ? S.val[slot][i] : 1.0f;
                            wv[q] = S.wp[slot][i];
                            lk[q] = S.link[slot][i];
                            acc = __fmaf_rn(wv[q], xv[q], acc);
                        }
                    }
                    const float m = warp_combine(acc);
                    const float c = __fmul_rn(eta, dev_grad(loss, m, S.y[slot]));
#pragma unroll
                    for (int q = 0; q < R; ++q) {
                        const int i = q * 32 + lane;
                        if (i < k) {
                            const float nw = __fsub_rn(wv[q], __fmul_rn(c, xv[q]));
                            S.out[slot][i] = nw;
                            if (lk[q] & LK_PUSH)
                                S.wp[(r + (int)((lk[q] >> 16) & 0xffu)) & (CH_SLOTS - 1)][lk[q] & 0xffffu] = nw;
                        }
                    }
                    __syncwarp();
                }
            }
            __syncthreads();
        }
        cp_wait_all();
        __syncthreads();
    }
}

// link[p] (layout above): receive flag from the previous occurrence, push
// target from the next occurrence, each when it lies within CH_D examples
__global__ void k_chain_link(const int32_t *__restrict__ prev, const int32_t *__restrict__ next,
                             const int32_t *__restrict__ row_of, const int64_t *__restrict__ row_ptr, int64_t nnz,
                             uint32_t *__restrict__ link, const int *status)
{
    if (read_status(status)) return;
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < nnz; p += (int64_t)gridDim.x * blockDim.x) {
        const int32_t t = row_of[p], q = prev[p], n = next[p];
        uint32_t l = 0;
        if (q >= 0 && t - row_of[q] <= CH_D) l |= LK_RECV;
        if (n >= 0) {
            const int32_t tn = row_of[n];
            if (tn - t <= CH_D) l |= LK_PUSH | ((uint32_t)(tn - t) << 16) | (uint32_t)(n - row_ptr[tn]);
        }
        link[p] = l;
    }
}

}  // namespace

namespace pdb {

int chain_max_row() { return CH_MAXK; }

int chain_schedule(const int32_t *prev, const int32_t *next, const int32_t *row_of, const int64_t *row_ptr,
                   int64_t nnz, uint32_t *link, const int *status, cudaStream_t s)
{
    if (nnz > 0) {
        k_chain_link<<<grid_1d(nnz), 256, 0, s>>>(prev, next, row_of, row_ptr, nnz, link, status);
        note_launch();
    }
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

int chain_run(const pdb_csr *X, const float *y, const uint32_t *link, float *w, int loss, float eta, int epochs,
              int max_row, int *status, cudaStream_t s)
{
    // registers per lane for the longest example: 1, 2, 4 or 8 (32 to 256 ids)
    auto kern = max_row <= 32 ? k_sgd_chain<1> : max_row <= 64 ? k_sgd_chain<2>
              : max_row <= 128 ? k_sgd_chain<4> : k_sgd_chain<8>;
    const int variant = max_row <= 32 ? 0 : max_row <= 64 ? 1 : max_row <= 128 ? 2 : 3;
    static bool configured[64][4] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !configured[dev][variant]) {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sizeof(ChainSmem)) !=
            cudaSuccess)
            return PDB_ECUDA;
        configured[dev][variant] = true;
    }
    kern<<<1, CH_THREADS, sizeof(ChainSmem), s>>>((int32_t)X->n_rows, X->row_ptr, X->col, X->val, y, link, w, loss,
                                                  eta, epochs, status);
    note_launch();
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

}  // namespace pdb
