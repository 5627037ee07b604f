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
//   warps 1-3, 5 prefetch one example of a step each with cp.async (ids,
//                values, labels and link words 4 steps ahead; the weights
//                nobody will push 2 steps ahead, together with the shared
//                memory address each new weight goes to), lanes striding
//                over the example's elements;
//   warps 6, 7   write the new weights of the previous step that are not
//                pushed through to global memory, and copy row bounds 7
//                steps ahead;
//   warp 4       only joins the barriers: warps map to the SM's four
//                schedulers by index mod 4, and warp 0 keeps its own.
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

#include <atomic>

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
// link word of a position: bit 31 = its weight will be pushed by an earlier
// example (skip the gather); bit 30 = push the new weight to the next
// occurrence, which is element (bits 0..7) of the example (bits 16..23)
// examples later; bit 29 = the previous occurrence is in the example just
// before, as its element (bits 8..15)
constexpr uint32_t LK_RECV = 1u << 31, LK_PUSH = 1u << 30, LK_LATE = 1u << 29;
static_assert((CH_SLOTS & (CH_SLOTS - 1)) == 0 && (CH_RP & (CH_RP - 1)) == 0, "ring sizes must be powers of two");
static_assert(CH_SLOTS > (CH_DS + 2) * CH_G && CH_RP > (CH_L + 2) * CH_G + 1, "rings too short");
static_assert(CH_D < 256 && CH_MAXK <= 256, "link word fields");
// store address word the compute warp reads per element: the shared-memory
// address of the new weight (below 2^22), bit 22 = the weight arrives from
// the example just before, as its element (bits 23..30)
constexpr uint32_t PA_ADDR = (1u << 22) - 1, PA_LATE = 1u << 22;
static_assert((CH_G & (CH_G - 1)) == 0, "examples per step must be a power of two");
// a weight is gathered (not pushed) when its last writer r' lies more than
// CH_D examples back; r' stores it through at step r'/G + 1, the gather for r
// runs at step r/G - CH_BS, and r/G - r'/G >= (CH_D + 1) / G: the store must
// land at least one step (one __syncthreads) before the gather
static_assert((CH_D + 1) / CH_G >= CH_BS + 2, "a gather may not meet its last writer's store in one step");

// ids and link words are copied in 16-byte pieces from the aligned element
// before the example's first one: element i sits at index off + i, off =
// (first position) mod 4 (0 when an input array is not 16-byte aligned).
// Everything the compute warp reads is at element index i, so its loads need
// no row bounds.
constexpr int CH_ROW = CH_MAXK + 4;
struct ChainSmem {
    int32_t col[CH_SLOTS][CH_ROW];
    uint32_t link[CH_SLOTS][CH_ROW];
    float xa[CH_SLOTS][CH_MAXK];    // value of each element (1 without values)
    uint32_t pa[CH_SLOTS][CH_MAXK]; // where the compute warp stores each element's new weight
    float wp[CH_SLOTS][CH_MAXK];    // weight each element reads (gathered or pushed)
    float out[CH_SLOTS][CH_MAXK];   // weight of the elements whose next occurrence is not pushed
    int64_t rp[CH_RP];
    float y[CH_SLOTS];
    int kk[CH_SLOTS];               // length of each example
    float dump[32];                 // store target of the lanes past an example's end
    __align__(16) float part[32];   // the compute warp's 32 partial sums
};

// The xor-butterfly combine of warp_combine (for off = 16, 8, 4, 2, 1 every
// lane adds the partial of lane ^ off), evaluated from shared memory: every
// lane reads the 32 partials and adds them in the same tree -- level by
// level, partial l plus partial l + half -- which is the value lane 0 ends
// with after the shuffles (fp32 addition is commutative, so every lane of
// the shuffle version holds it too).  Two shared-memory round trips instead
// of five dependent shuffles.
__device__ __forceinline__ float combine_smem(float a, float *part)
{
    part[threadIdx.x & 31] = a;
    __syncwarp();
    float v[32];
    const float4 *p4 = reinterpret_cast<const float4 *>(part);
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        const float4 f = p4[q];
        v[4 * q] = f.x;
        v[4 * q + 1] = f.y;
        v[4 * q + 2] = f.z;
        v[4 * q + 3] = f.w;
    }
#pragma unroll
    for (int half = 16; half >= 1; half >>= 1)
#pragma unroll
        for (int l = 0; l < half; ++l) v[l] = __fadd_rn(v[l], v[l + half]);
    return v[0];
}

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
__device__ __forceinline__ void cp16(void *smem_dst, const void *gsrc)
{
    const unsigned d = (unsigned)__cvta_generic_to_shared(smem_dst);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(gsrc) : "memory");
}
// copies elements [a0, b + k) of a 4-byte array into dst[0 ..): with vec
// (every source array 16-byte aligned) in 16-byte pieces from the aligned
// a0 = b - off up to the last aligned position and then the tail one element
// at a time; without, all of it one element at a time (off = 0)
__device__ __forceinline__ void cp_row(void *dst, const void *src, int64_t b, int k, int off, bool vec, int lane)
{
    const int64_t a0 = b - off;
    const int64_t a1 = vec ? ((b + k) & ~(int64_t)3) : a0;
    const int n16 = a1 > a0 ? (int)((a1 - a0) >> 2) : 0;
    for (int c = lane; c < n16; c += 32)
        cp16((uint32_t *)dst + 4 * c, (const uint32_t *)src + a0 + 4 * c);
    for (int64_t e = (a1 > b ? a1 : b) + lane; e < b + k; e += 32)
        cp4((uint32_t *)dst + (e - a0), (const uint32_t *)src + e);
}
__device__ __forceinline__ void st_shared(unsigned addr, float v)
{
    asm volatile("st.shared.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_wait_b() { asm volatile("cp.async.wait_group %0;" ::"n"(CH_BS - 1) : "memory"); }
__device__ __forceinline__ void cp_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// bounds [b, b + k) of example r from the row_ptr ring (false outside
// 0..N-1) and the offset of its elements in the 16-byte-copied rows
__device__ __forceinline__ bool row_bounds(const ChainSmem &S, int r, int N, bool vec, int64_t &b, int &k, int &off)
{
    if (r < 0 || r >= N) return false;
    b = S.rp[r & (CH_RP - 1)];
    k = (int)(S.rp[(r + 1) & (CH_RP - 1)] - b);
    off = vec ? (int)(b & 3) : 0;
    return true;
}

template <int R, int LOSS>
__global__ __launch_bounds__(CH_THREADS, 1) void k_sgd_chain(int32_t n_rows, const int64_t *__restrict__ row_ptr,
                                                             const int32_t *__restrict__ col,
                                                             const float *__restrict__ val,
                                                             const float *__restrict__ y,
                                                             const uint32_t *__restrict__ link, float *w, int loss,
                                                             float eta, int epochs, bool vec, int *status,
                                                             uint64_t *trace)
{
    extern __shared__ __align__(16) unsigned char smem_raw[];
    ChainSmem &S = *reinterpret_cast<ChainSmem *>(smem_raw);
    if (read_status(status)) return;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // warp 0 computes; warps 1, 2, 3, 5 prefetch example g = 0..3 of a step
    // (ids, values, link words, then weights and store addresses); warps 6, 7
    // write the weights of the previous step through (two examples each) and
    // copy row bounds; warp 4 only joins the barriers (it shares warp 0's
    // scheduler)
    const bool compute = warp == 0;
    const unsigned wp_base = (unsigned)__cvta_generic_to_shared(&S.wp[0][0]);
    const unsigned out_base = (unsigned)__cvta_generic_to_shared(&S.out[0][0]);
    const int gA = warp >= 1 && warp <= 3 ? warp - 1 : warp == 5 ? 3 : -1;
    const int gW = warp == 6 ? 0 : warp == 7 ? 2 : -1;
    const int N = n_rows;
    const int steps = (N + CH_G - 1) / CH_G;

    for (int ep = 0; ep < epochs; ++ep) {
        for (int t = -CH_L; t <= steps; ++t) {
            if (gW >= 0) {
                // stage W: new weights of step t - 1 that no example among the next D takes
                // on chip go through to global memory (a pushed weight is re-written by its
                // receiver, so two stores of one step never hit one address)
                for (int g = gW; g < gW + 2; ++g) {
                    const int r = (t - 1) * CH_G + g;
                    int64_t b;
                    int k, off;
                    if (row_bounds(S, r, N, vec, b, k, off)) {
                        const int slot = r & (CH_SLOTS - 1);
                        for (int i = lane; i < k; i += 32)
                            if (!(S.link[slot][off + i] & LK_PUSH)) w[S.col[slot][off + i]] = S.out[slot][i];
                    }
                }
                // stage R: row_ptr entries [(t+L)G, (t+L)G + G) with L = DS + BS + 1, so that
                // stage A of step t finds the bounds of step t + DS (and the entry after it) complete
                if (warp == 6 && lane < CH_G) {
                    const int r = (t + CH_L) * CH_G + lane;
                    if (r >= 0 && r <= N) cp8(&S.rp[r & (CH_RP - 1)], row_ptr + r);
                }
            } else if (gA >= 0) {
                // stage A: ids, values, link words and label of example g of step t + DS
                {
                    const int r = (t + CH_DS) * CH_G + gA;
                    int64_t b;
                    int k, off;
                    if (row_bounds(S, r, N, vec, b, k, off)) {
                        const int slot = r & (CH_SLOTS - 1);
                        cp_row(S.col[slot], col, b, k, off, vec, lane);
                        cp_row(S.link[slot], link, b, k, off, vec, lane);
                        for (int i = lane; i < k; i += 32) {
                            if (val)
                                cp4(&S.xa[slot][i], val + b + i);
                            else
                                S.xa[slot][i] = 1.0f;
                        }
                        if (lane == 0) cp4(&S.y[slot], y + r);
                    }
                }
                // stage B: weights of example g of step t + BS that no recent example pushes,
                // and where the compute warp stores each element's new weight: into the
                // receiver's slot of wp when pushed, else into out (written through by 6, 7)
                {
                    const int r = (t + CH_BS) * CH_G + gA;
                    int64_t b;
                    int k, off;
                    if (row_bounds(S, r, N, vec, b, k, off)) {
                        const int slot = r & (CH_SLOTS - 1);
                        for (int i = lane; i < k; i += 32) {
                            const uint32_t lk = S.link[slot][off + i];
                            if (!(lk & LK_RECV)) cp4(&S.wp[slot][i], w + S.col[slot][off + i]);
                            const unsigned tslot = ((unsigned)r + ((lk >> 16) & 0xffu)) & (CH_SLOTS - 1);
                            const unsigned addr = (lk & LK_PUSH) ? wp_base + 4u * (tslot * CH_MAXK + (lk & 0xffu))
                                                                 : out_base + 4u * ((unsigned)slot * CH_MAXK + i);
                            S.pa[slot][i] = addr | ((lk & LK_LATE) ? PA_LATE | (((lk >> 8) & 0xffu) << 23) : 0u);
                        }
                        if (lane == 0) S.kk[slot] = k;
                    }
                }
            }
            if (!compute) {
                cp_commit();
                cp_wait_b();
            } else if (t >= 0 && t < steps) {
                // compute the G examples of step t in data order.  The first takes every
                // weight from its slot.  Each later one fetches its length, label, values,
                // store words and weights while the example before computes its gradient:
                // a weight that example writes (its previous occurrence is there) is taken
                // from it once it exists -- by shuffle from the lane that computed it for
                // rows of up to 64 ids, else from the slot after the pushes are stored --
                // and every other weight is final when fetched.
                const int r0 = t * CH_G, r1 = min(N, r0 + CH_G);
                const unsigned dump = (unsigned)__cvta_generic_to_shared(&S.dump[lane]);
                int k;
                float yr, xv[R], wv[R];
                unsigned pa[R];
                auto fetch = [&](int r) {
                    const int slot = r & (CH_SLOTS - 1);
                    k = S.kk[slot];
                    yr = S.y[slot];
#pragma unroll
                    for (int q = 0; q < R; ++q) {
                        xv[q] = S.xa[slot][q * 32 + lane];
                        pa[q] = S.pa[slot][q * 32 + lane];
                        wv[q] = S.wp[slot][q * 32 + lane];      // past k: unused
                    }
                };
                fetch(r0);
                for (int r = r0; r < r1; ++r) {
                    float wc[R], xc[R], nw[R];
                    unsigned ac[R];
                    float acc = 0.0f;
#pragma unroll
                    for (int q = 0; q < R; ++q) {
                        const int i = q * 32 + lane;
                        wc[q] = wv[q];
                        xc[q] = xv[q];
                        const float f = __fmaf_rn(wc[q], xc[q], acc);
                        acc = i < k ? f : acc;
                        ac[q] = i < k ? (pa[q] & PA_ADDR) : dump;
                    }
                    const float yc = yr;
                    trace_mark(trace, (int64_t)ep * N + r, 0);    // every weight is read
                    const float m = combine_smem(acc, S.part);
                    if (r + 1 < r1) fetch(r + 1);
                    const float c = __fmul_rn(eta, dev_grad(LOSS, m, yc));
                    trace_mark(trace, (int64_t)ep * N + r, 1);   // before any write is visible
#pragma unroll
                    for (int q = 0; q < R; ++q) {
                        nw[q] = __fsub_rn(wc[q], __fmul_rn(c, xc[q]));
                        st_shared(ac[q], nw[q]);
                    }
                    __syncwarp();
                    if (r + 1 < r1) {
                        const int nslot = (r + 1) & (CH_SLOTS - 1);
#pragma unroll
                        for (int q = 0; q < R; ++q) {
                            const unsigned src = (pa[q] >> 23) & 0xffu;   // element of r
                            if (R <= 2) {
                                float v = wv[q];
#pragma unroll
                                for (int qs = 0; qs < R; ++qs) {
                                    const float u = __shfl_sync(FULL, nw[qs], (int)(src & 31u));
                                    if ((pa[q] & PA_LATE) && (int)(src >> 5) == qs) v = u;
                                }
                                wv[q] = v;
                            } else if (pa[q] & PA_LATE) {
                                wv[q] = S.wp[nslot][q * 32 + lane];   // stored above, before the __syncwarp
                            }
                        }
                    }
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
        if (q >= 0 && row_of[q] == t - 1) l |= LK_LATE | ((uint32_t)(q - row_ptr[t - 1]) << 8);
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

using ChainKernel = void (*)(int32_t, const int64_t *, const int32_t *, const float *, const float *,
                             const uint32_t *, float *, int, float, int, bool, int *, uint64_t *);

template <int R>
static ChainKernel chain_kernel(int loss)
{
    return loss == PDB_LOSS_LOGISTIC ? k_sgd_chain<R, PDB_LOSS_LOGISTIC>
           : loss == PDB_LOSS_SQUARED ? k_sgd_chain<R, PDB_LOSS_SQUARED> : k_sgd_chain<R, PDB_LOSS_HINGE>;
}

int chain_run(const pdb_csr *X, const float *y, const uint32_t *link, float *w, int loss, float eta, int epochs,
              int max_row, int *status, uint64_t *trace, cudaStream_t s)
{
    // registers per lane for the longest example: 1, 2, 4 or 8 (32 to 256 ids);
    // one kernel per loss, so the gradient has no branch
    const int rw = max_row <= 32 ? 0 : max_row <= 64 ? 1 : max_row <= 128 ? 2 : 3;
    const ChainKernel kern = rw == 0 ? chain_kernel<1>(loss) : rw == 1 ? chain_kernel<2>(loss)
                             : rw == 2 ? chain_kernel<4>(loss) : chain_kernel<8>(loss);
    const int variant = rw * 3 + (loss >= 0 && loss <= 2 ? loss : 2);
    // set once per device and variant (any device past the table: every call)
    static std::atomic<bool> configured[64][12];
    int dev = 0;
    cudaGetDevice(&dev);
    const bool known = dev >= 0 && dev < 64;
    if (!known || !configured[dev][variant].load(std::memory_order_acquire)) {
        if (cudaFuncSetAttribute((const void *)kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)sizeof(ChainSmem)) != cudaSuccess)
            return PDB_ECUDA;
        if (known) configured[dev][variant].store(true, std::memory_order_release);
    }
    // 16-byte row copies need 16-byte aligned ids, values and link words
    const bool vec = ((uintptr_t)X->col & 15) == 0 && ((uintptr_t)X->val & 15) == 0 && ((uintptr_t)link & 15) == 0;
    kern<<<1, CH_THREADS, sizeof(ChainSmem), s>>>((int32_t)X->n_rows, X->row_ptr, X->col, X->val, y, link, w, loss,
                                                  eta, epochs, vec, status, trace);
    note_launch();
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

}  // namespace pdb
