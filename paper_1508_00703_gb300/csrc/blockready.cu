// Block-resident ready-counter engine: pdb_sgd_epoch under a READY schedule
// when the per-feature (weight, version) records of all n_cols features fit
// in one thread block's shared memory (up to ~20,000 features).
//
// Same protocol as the grid-wide READY engine (the read protocol of Section
// 5 per feature; record = bits(w_j) | version << 32, versions carrying an
// epoch stamp so all epochs run in one launch), but the records live in
// shared memory: a wait is a shared-memory poll of a few tens of cycles
// instead of an L2 round trip, which is what bounds data with many short
// dependency hops (the tiny workload: 441 levels of ~45 examples).
//
// 32 warps take examples in data order (epoch-major) from a shared ticket
// counter.  Each warp keeps three examples in flight: the row bounds of the
// one after next and the ids, values and gate words of the next are loading
// while it waits on and computes the current one, so the two dependent
// global-memory latencies overlap earlier examples.  The oldest unfinished
// example never waits on a younger one (its predecessors hold smaller
// tickets and each warp finishes its examples in ticket order), so there is
// no deadlock; every wait is bounded.
#include <cuda_runtime.h>

#include "common.cuh"

using namespace pdb;

namespace {

constexpr int BR_THREADS = 1024;
constexpr int BR_R = 2;                 // elements per lane: rows of at most 64 ids

__device__ __forceinline__ unsigned long long ld_srec(const unsigned long long *p)
{
    unsigned long long v;
    asm volatile("ld.relaxed.cta.shared.b64 %0, [%1];" : "=l"(v) : "r"((unsigned)__cvta_generic_to_shared(p)) : "memory");
    return v;
}
__device__ __forceinline__ void st_srec(unsigned long long *p, float w, unsigned version)
{
    const unsigned long long v = (unsigned long long)__float_as_uint(w) | ((unsigned long long)version << 32);
    asm volatile("st.relaxed.cta.shared.b64 [%0], %1;" ::"r"((unsigned)__cvta_generic_to_shared(p)), "l"(v) : "memory");
}

__device__ __forceinline__ unsigned stamp_of(int64_t e) { return (1u + (unsigned)(e % 7)) << 29; }

// tg / n exactly (tickets below 2^31 here): a float estimate, then integer
// corrections -- cheaper than a 64-bit division on the per-example path
__device__ __forceinline__ int epoch_of(int64_t tg, int32_t n, float inv_n)
{
    int e = __float2int_rz((float)tg * inv_n);
    while (e > 0 && (int64_t)e * n > tg) --e;
    while ((int64_t)(e + 1) * n <= tg) ++e;
    return e;
}

// one example's inputs, loaded ahead
struct Ex {
    int64_t tg;         // ticket (example index over all epochs), -1 = none
    int epoch;
    int k;
    float y;
    int j[BR_R];
    float x[BR_R];
    uint32_t g[BR_R];
};

// row bounds of ticket tg (example tg mod n_rows), issued two examples ahead
struct Bounds {
    int64_t tg, b, e;
    int epoch, t;
};
__device__ __forceinline__ void load_bounds(Bounds &B, int64_t tg, int64_t total, int32_t n_rows, float inv_n,
                                            const int64_t *__restrict__ row_ptr)
{
    B.tg = tg < total ? tg : -1;
    B.b = B.e = 0;
    B.epoch = B.t = 0;
    if (B.tg < 0) return;
    B.epoch = epoch_of(tg, n_rows, inv_n);
    B.t = (int)(tg - (int64_t)B.epoch * n_rows);
    B.b = row_ptr[B.t];
    B.e = row_ptr[B.t + 1];
}

// ids, values, gate words and label of the example whose bounds are B, one example ahead
__device__ __forceinline__ void load_ex(Ex &e, const Bounds &B, int32_t n_rows, const int32_t *__restrict__ col,
                                        const float *__restrict__ val, const float *__restrict__ y,
                                        const uint32_t *__restrict__ gate, int lane)
{
    e.tg = B.tg;
    e.epoch = B.epoch;
    e.k = (int)(B.e - B.b);
    e.y = B.tg >= 0 ? y[B.t] : 0.0f;
#pragma unroll
    for (int r = 0; r < BR_R; ++r) {
        const int i = r * 32 + lane;
        e.j[r] = i < e.k ? col[B.b + i] : 0;
        e.x[r] = i < e.k ? (val ? val[B.b + i] : 1.0f) : 0.0f;
        e.g[r] = i < e.k ? gate[B.b + i] : 0u;
    }
}

__global__ __launch_bounds__(BR_THREADS, 1) void k_sgd_block_ready(int32_t n_rows, int64_t n_cols,
                                                                   const int64_t *__restrict__ row_ptr,
                                                                   const int32_t *__restrict__ col,
                                                                   const float *__restrict__ val,
                                                                   const float *__restrict__ y,
                                                                   const uint32_t *__restrict__ gate, float *w,
                                                                   int loss, float eta, int epochs, int *status,
                                                                   uint64_t timeout, uint64_t *trace)
{
    extern __shared__ __align__(16) unsigned char smem_raw[];
    unsigned long long *rec = reinterpret_cast<unsigned long long *>(smem_raw);
    __shared__ unsigned long long ticket;
    if (read_status(status)) return;
    const int lane = threadIdx.x & 31;
    for (int64_t f = threadIdx.x; f < n_cols; f += BR_THREADS)
        rec[f] = (unsigned long long)__float_as_uint(w[f]) | ((unsigned long long)stamp_of(0) << 32);
    if (threadIdx.x == 0) ticket = 0;
    __syncthreads();

    const int64_t total = (int64_t)epochs * n_rows;
    auto take = [&]() -> int64_t {
        unsigned long long tk = 0;
        if (lane == 0) tk = atomicAdd(&ticket, 1ull);
        return (int64_t)__shfl_sync(FULL, tk, 0);
    };
    // three examples in flight per warp: bounds two ahead, data one ahead
    Ex cur, nxt;
    Bounds bc, bn;
    const float inv_n = 1.0f / (float)n_rows;
    load_bounds(bc, take(), total, n_rows, inv_n, row_ptr);
    load_bounds(bn, take(), total, n_rows, inv_n, row_ptr);
    load_ex(cur, bc, n_rows, col, val, y, gate, lane);
    bool failed = false;
    while (cur.tg >= 0) {
        Bounds bnn;
        load_bounds(bnn, take(), total, n_rows, inv_n, row_ptr);
        load_ex(nxt, bn, n_rows, col, val, y, gate, lane);      // in flight while cur runs
        bn = bnn;
        const unsigned stamp = stamp_of(cur.epoch), next_stamp = stamp_of(cur.epoch + 1);
        float wv[BR_R];
        unsigned pending = 0;
#pragma unroll
        for (int r = 0; r < BR_R; ++r) {
            wv[r] = 0.0f;
            if (r * 32 + lane < cur.k) {
                const unsigned long long v = ld_srec(rec + cur.j[r]);
                wv[r] = __uint_as_float((unsigned)v);
                if ((unsigned)(v >> 32) != ((cur.g[r] & GATE_RANK) | stamp)) pending |= 1u << r;
            }
        }
        if (pending) {
            const uint64_t t0 = globaltimer();
            unsigned spins = 0;
            while (pending && !failed) {
#pragma unroll
                for (int r = 0; r < BR_R; ++r)
                    if (pending & (1u << r)) {
                        const unsigned long long v = ld_srec(rec + cur.j[r]);
                        if ((unsigned)(v >> 32) == ((cur.g[r] & GATE_RANK) | stamp)) {
                            wv[r] = __uint_as_float((unsigned)v);
                            pending &= ~(1u << r);
                        }
                    }
                if (pending) __nanosleep(32);   // leave issue slots to the warps that can run
                if (pending && (++spins & 63u) == 0) {
                    if (read_status(status)) failed = true;
                    else if (globaltimer() - t0 > timeout) {
                        set_status(status, PDB_ETIMEOUT);
                        failed = true;
                    }
                }
            }
        }
        if (__any_sync(FULL, failed)) break;     // every warp still reaches the barrier below
        trace_mark(trace, cur.tg, 0);
        float acc = 0.0f;
#pragma unroll
        for (int r = 0; r < BR_R; ++r)
            if (r * 32 + lane < cur.k) acc = __fmaf_rn(wv[r], cur.x[r], acc);
        const float m = warp_combine(acc);
        const float c = __fmul_rn(eta, dev_grad(loss, m, cur.y));
        trace_mark(trace, cur.tg, 1);   // before any write is visible
#pragma unroll
        for (int r = 0; r < BR_R; ++r)
            if (r * 32 + lane < cur.k) {
                const uint32_t g = cur.g[r];
                st_srec(rec + cur.j[r], __fsub_rn(wv[r], __fmul_rn(c, cur.x[r])),
                        (g & GATE_LAST) ? next_stamp : ((g & GATE_RANK) + 1u) | stamp);
            }
        cur = nxt;
    }
    __syncthreads();
    for (int64_t f = threadIdx.x; f < n_cols; f += BR_THREADS) w[f] = __uint_as_float((unsigned)rec[f]);
}

}  // namespace

namespace pdb {

// shared memory for the block-resident READY engine, 0 when it does not apply
int64_t block_ready_smem(int64_t n_cols, int64_t max_row)
{
    if (n_cols < 1 || max_row > 32 * BR_R) return 0;
    int dev = 0, optin = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    const int64_t bytes = n_cols * 8;
    return bytes + 1024 <= optin ? bytes : 0;
}

int block_ready_run(const pdb_csr *X, const float *y, const uint32_t *gate, float *w, int loss, float eta,
                    int epochs, int max_row, int *status, uint64_t timeout, uint64_t *trace, cudaStream_t s)
{
    const int64_t smem = block_ready_smem(X->n_cols, max_row);
    if (smem == 0) return PDB_ETOOBIG;
    if (cudaFuncSetAttribute(k_sgd_block_ready, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
        cudaSuccess)
        return PDB_ECUDA;
    k_sgd_block_ready<<<1, BR_THREADS, (size_t)smem, s>>>((int32_t)X->n_rows, X->n_cols, X->row_ptr, X->col,
                                                          X->val, y, gate, w, loss, eta, epochs, status, timeout, trace);
    note_launch();
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

}  // namespace pdb
