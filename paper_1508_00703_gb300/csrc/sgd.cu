// Update engines: pdb_sgd_epoch's level-synchronous and ready-counter
// dataflow engines and its dispatch to the others (window.cu, blockready.cu,
// chain.cu, resident.cu); the host side of pdb_ssp_epoch (kernels in
// ssp.cu); pdb_bsp_epoch (the BSP mini-batch comparison).
//
// In the two engines here one warp runs one example (one transaction,
// Definition 3): the lanes load the example's ids and values with coalesced
// loads, gather w through L2, form the margin with per-lane fused
// multiply-adds and a xor-shuffle combine, compute the scalar eta*g, and
// scatter w_j -= eta*g*x_j.  No atomics touch w: the schedule guarantees
// that no other example holds any of these features at the same time.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <new>
#include <mutex>

#include "common.cuh"

using namespace pdb;

namespace {



// ---------------------------------------------------------------- one example, no waits
// Used by the level-synchronous engine: the level schedule already keeps
// every example of a level disjoint from the others (Theorem 3).  Element i
// of the row lives in lane i mod 32, register i / 32; each lane accumulates
// its elements in increasing i with fused multiply-adds, then the lanes
// combine pairwise (the fixed order both sides of the parity check use).
template <int R>
__device__ __forceinline__ void sgd_example(int t, const int64_t *__restrict__ row_ptr, const int32_t *__restrict__ col,
                                            const float *__restrict__ val, const float *__restrict__ y, float *w,
                                            int loss, float eta, uint64_t *trace, int64_t idx)
{
    const int lane = threadIdx.x & 31;
    const int64_t b = row_ptr[t];
    const int k = (int)(row_ptr[t + 1] - b);
    const float yt = y[t];
    float acc = 0.0f;
    if (k <= 32 * R) {
        int j[R];
        float x[R], wv[R];
#pragma unroll
        for (int r = 0; r < R; ++r) {
            int i = r * 32 + lane;
            j[r] = i < k ? col[b + i] : 0;
            x[r] = i < k ? (val ? val[b + i] : 1.0f) : 0.0f;
        }
#pragma unroll
        for (int r = 0; r < R; ++r)
            if (r * 32 + lane < k) wv[r] = __ldcg(w + j[r]);
#pragma unroll
        for (int r = 0; r < R; ++r)
            if (r * 32 + lane < k) acc = __fmaf_rn(wv[r], x[r], acc);
        const float m = warp_combine(acc);       // every lane's loads have returned
        trace_mark(trace, idx, 0);
        const float c = __fmul_rn(eta, dev_grad(loss, m, yt));
        trace_mark(trace, idx, 1);   // before any write is visible
#pragma unroll
        for (int r = 0; r < R; ++r)
            if (r * 32 + lane < k) __stcg(w + j[r], __fsub_rn(wv[r], __fmul_rn(c, x[r])));
    } else {
        for (int i = lane; i < k; i += 32) acc = __fmaf_rn(__ldcg(w + col[b + i]), val ? val[b + i] : 1.0f, acc);
        const float m = warp_combine(acc);
        trace_mark(trace, idx, 0);
        const float c = __fmul_rn(eta, dev_grad(loss, m, yt));
        trace_mark(trace, idx, 1);   // before any write is visible
        for (int i = lane; i < k; i += 32) {
            int jj = col[b + i];
            float xx = val ? val[b + i] : 1.0f;
            __stcg(w + jj, __fsub_rn(__ldcg(w + jj), __fmul_rn(c, xx)));
        }
    }
    __syncwarp();
}

// ---------------------------------------------------------------- level-synchronous engine
// Persistent cooperative kernel: level l's examples are spread over all
// warps, a grid barrier closes the level (the read barrier of the next BSP
// step and the write barrier of this one, Algorithm 2a per level).
template <int R>
__global__ __launch_bounds__(THREADS) void k_sgd_levels(int32_t n_rows, const int64_t *__restrict__ row_ptr,
                                                        const int32_t *__restrict__ col, const float *__restrict__ val,
                                                        const float *__restrict__ y, const int32_t *__restrict__ order,
                                                        const int64_t *__restrict__ level_ptr, const LevelCtl *ctl,
                                                        float *w, int loss, float eta, int epochs, GridBarrier *bar,
                                                        int *status, uint64_t timeout, uint64_t *trace)
{
    if (read_status(status)) return;
    const int L = ctl->n_levels;
    const int gw = (int)(((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
    const int nw = (int)(((int64_t)gridDim.x * blockDim.x) >> 5);
    for (int ep = 0; ep < epochs; ++ep)
        for (int l = 0; l < L; ++l) {
            const int64_t b = level_ptr[l], e = level_ptr[l + 1];
            for (int64_t i = b + gw; i < e; i += nw) {
                const int t = order[i];
                if (t < 0 || t >= n_rows) {      // cannot happen with a consistent schedule
                    set_status(status, PDB_EFAULT);
                    continue;
                }
                sgd_example<R>(t, row_ptr, col, val, y, w, loss, eta, trace, (int64_t)ep * n_rows + t);
            }
            if (!grid_sync(bar, status, timeout)) return;
        }
}

// ---------------------------------------------------------------- ready-counter dataflow engine
// The read protocol of Section 5 per feature.  Feature j's record holds its
// weight and its iteration number (version) in one aligned 64-bit word:
// rec[j] = bits(w_j) | version_j << 32.  The occurrence of j with rank r
// (its gate) may read w_j once version_j == r -- one relaxed 64-bit load
// both checks the version and returns the weight written with it (Read
// Constraint: the previous writer is done) -- and publishes the new weight
// together with version r + 1 in one 64-bit store (Write Constraint: its own
// read, the only read of that version, came first).  Both halves travel in
// one single-copy-atomic access, so no fence is needed.
// All epochs run in one launch, pipelined: a version carries the epoch's
// stamp (1..7, bits 29-31 above the 29-bit rank), and the last occurrence
// of j in an epoch (GATE_LAST) publishes version 0 with the next epoch's
// stamp, so the next epoch's first occurrence of j starts as soon as that
// write lands -- not at a kernel boundary (exact by Theorem 2: per feature
// the order is still the data order, epoch after epoch).  A record only
// ever holds a version of the current or the previous epoch of its
// feature, so stamps that repeat every 7 epochs never match stale ones.
// Examples are taken in data order (epoch-major) from a ticket counter,
// `chunk` consecutive ones at a time and run in order by the warp that took
// them, so the oldest unfinished example never waits on a younger one and
// the kernel cannot deadlock whatever the number of resident warps.
__device__ __forceinline__ unsigned long long ld_rec(const unsigned long long *p)
{
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_rec(unsigned long long *p, float w, unsigned version)
{
    unsigned long long v = (unsigned long long)__float_as_uint(w) | ((unsigned long long)version << 32);
    asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

// Gathers w for the lane's elements, waiting until each record carries the
// wanted version.  False when the wait gave up (timeout or a failure
// elsewhere recorded in status).
template <int R>
__device__ __forceinline__ bool gather_ready(const unsigned long long *rec, const int *j, const unsigned *want,
                                             float *wv, int lane, int k, int *status, uint64_t timeout)
{
    unsigned pending = 0;
#pragma unroll
    for (int r = 0; r < R; ++r)
        if (r * 32 + lane < k) {
            unsigned long long v = ld_rec(rec + j[r]);
            wv[r] = __uint_as_float((unsigned)v);
            if ((unsigned)(v >> 32) != want[r]) pending |= 1u << r;
        }
    if (pending == 0) return true;
    const uint64_t t0 = globaltimer();
    unsigned spins = 0, nap = 32;
    while (pending) {
        // back off so a waiting lane does not flood L2 with polls; the cap
        // (128 ns) is the latency of a hop on mid-conflict data, where READY
        // is AUTO's choice (512 ns was 16% slower on the tiny workload)
        __nanosleep(nap);
        nap = nap < 128 ? 2 * nap : 128;
#pragma unroll
        for (int r = 0; r < R; ++r)
            if (pending & (1u << r)) {
                unsigned long long v = ld_rec(rec + j[r]);
                if ((unsigned)(v >> 32) == want[r]) {
                    wv[r] = __uint_as_float((unsigned)v);
                    pending &= ~(1u << r);
                }
            }
        if (pending && (++spins & 15u) == 0) {
            if (read_status(status)) return false;
            if (globaltimer() - t0 > timeout) {
                set_status(status, PDB_ETIMEOUT);
                return false;
            }
        }
    }
    return true;
}

// one example under the ready protocol; false when a wait gave up
__host__ __device__ __forceinline__ unsigned epoch_stamp(int64_t e) { return (1u + (unsigned)(e % 7)) << 29; }

template <int R>
__device__ __forceinline__ bool ready_example(int t, unsigned stamp, unsigned next_stamp,
                                              const int64_t *__restrict__ row_ptr,
                                              const int32_t *__restrict__ col, const float *__restrict__ val,
                                              const float *__restrict__ y, const uint32_t *__restrict__ gate,
                                              unsigned long long *rec, int loss, float eta, int *status,
                                              uint64_t timeout, uint64_t *trace, int64_t idx)
{
    const int lane = threadIdx.x & 31;
    const int64_t b = row_ptr[t];
    const int k = (int)(row_ptr[t + 1] - b);
    const float yt = y[t];
    if (k <= 32 * R) {
        int j[R];
        float x[R], wv[R];
        unsigned want[R], next[R];
#pragma unroll
        for (int r = 0; r < R; ++r) {
            int i = r * 32 + lane;
            j[r] = i < k ? col[b + i] : 0;
            x[r] = i < k ? (val ? val[b + i] : 1.0f) : 0.0f;
            uint32_t g = i < k ? gate[b + i] : 0u;
            want[r] = (g & GATE_RANK) | stamp;
            next[r] = (g & GATE_LAST) ? next_stamp : want[r] + 1u;
            wv[r] = 0.0f;
        }
        bool ok = gather_ready<R>(rec, j, want, wv, lane, k, status, timeout);
        if (!__all_sync(FULL, ok)) return false;
        trace_mark(trace, idx, 0);
        float acc = 0.0f;
#pragma unroll
        for (int r = 0; r < R; ++r)
            if (r * 32 + lane < k) acc = __fmaf_rn(wv[r], x[r], acc);
        const float m = warp_combine(acc);
        const float c = __fmul_rn(eta, dev_grad(loss, m, yt));
        trace_mark(trace, idx, 1);   // before any write is visible
#pragma unroll
        for (int r = 0; r < R; ++r)
            if (r * 32 + lane < k) st_rec(rec + j[r], __fsub_rn(wv[r], __fmul_rn(c, x[r])), next[r]);
        return true;
    }
    // long example: wait and gather element by element, then a second pass
    // (this example owns its features until it writes them, so re-reading
    // the records returns the same weights)
    float acc = 0.0f;
    bool ok = true;
    for (int i = lane; i < k && ok; i += 32) {
        int j1[1] = {col[b + i]};
        unsigned w1[1] = {(gate[b + i] & GATE_RANK) | stamp};
        float v1[1];
        ok = gather_ready<1>(rec, j1, w1, v1, 0, 1, status, timeout);
        if (ok) acc = __fmaf_rn(v1[0], val ? val[b + i] : 1.0f, acc);
    }
    if (!__all_sync(FULL, ok)) return false;
    trace_mark(trace, idx, 0);
    const float m = warp_combine(acc);
    const float c = __fmul_rn(eta, dev_grad(loss, m, yt));
    trace_mark(trace, idx, 1);   // before any write is visible
    for (int i = lane; i < k; i += 32) {
        const int jj = col[b + i];
        const float xx = val ? val[b + i] : 1.0f;
        const uint32_t g = gate[b + i];
        const float wo = __uint_as_float((unsigned)ld_rec(rec + jj));
        st_rec(rec + jj, __fsub_rn(wo, __fmul_rn(c, xx)), (g & GATE_LAST) ? next_stamp : ((g & GATE_RANK) + 1u) | stamp);
    }
    return true;
}

template <int R>
__global__ __launch_bounds__(THREADS) void k_sgd_ready(int32_t n_rows, const int64_t *__restrict__ row_ptr,
                                                       const int32_t *__restrict__ col, const float *__restrict__ val,
                                                       const float *__restrict__ y, const uint32_t *__restrict__ gate,
                                                       unsigned long long *rec, int loss, float eta, int epochs,
                                                       unsigned long long *ticket, int chunk, int *status,
                                                       uint64_t timeout, uint64_t *trace)
{
    if (read_status(status)) return;
    const int lane = threadIdx.x & 31;
    const int64_t total = (int64_t)epochs * n_rows;     // examples of all epochs, epoch-major
    for (;;) {
        unsigned long long tk = 0;
        if (lane == 0) tk = atomicAdd(ticket, (unsigned long long)chunk);
        tk = __shfl_sync(FULL, tk, 0);
        if (tk >= (unsigned long long)total) return;
        const int64_t t1 = min64(total, (int64_t)tk + chunk);
        for (int64_t tg = (int64_t)tk; tg < t1; ++tg) {
            const int64_t e = tg / n_rows;
            if (!ready_example<R>((int)(tg - e * n_rows), epoch_stamp(e), epoch_stamp(e + 1), row_ptr, col, val, y,
                                  gate, rec, loss, eta, status, timeout, trace, tg))
                return;
        }
    }
}

// rec[j] = (w_j, version 0 of the first epoch) before the first epoch; w_j
// back after the last
__global__ void k_pack(const float *__restrict__ w, int64_t n, unsigned long long *__restrict__ rec, const int *status)
{
    if (read_status(status)) return;
    const unsigned long long v0 = (unsigned long long)epoch_stamp(0) << 32;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        rec[i] = (unsigned long long)__float_as_uint(w[i]) | v0;
}

__global__ void k_unpack(const unsigned long long *__restrict__ rec, int64_t n, float *__restrict__ w,
                         const int *status)
{
    if (read_status(status)) return;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        w[i] = __uint_as_float((unsigned)rec[i]);
}

// ---------------------------------------------------------------- BSP
// margin of example t at the current w (all lanes return the same value)
__device__ __forceinline__ float margin(int t, const int64_t *__restrict__ row_ptr, const int32_t *__restrict__ col,
                                        const float *__restrict__ val, const float *w)
{
    const int lane = threadIdx.x & 31;
    const int64_t b = row_ptr[t];
    const int k = (int)(row_ptr[t + 1] - b);
    float acc = 0.0f;
    for (int i = lane; i < k; i += 32) acc = __fmaf_rn(__ldcg(w + col[b + i]), val ? val[b + i] : 1.0f, acc);
    return warp_combine(acc);
}

// The next CH terms of feature j's run from q (the batch's sorted pairs end at
// s1, its products start at s0), added to delta in ascending example order.
// Loads first, then the dependent adds.  Returns whether the run continues
// past the chunk (q then points after it).
template <int CH>
__device__ __forceinline__ bool run_chunk_prod(int32_t j, int64_t &q, int64_t s0, int64_t s1,
                                               const int32_t *__restrict__ bcol, const float *prod, float &delta)
{
    int32_t jj[CH];
    float pp[CH];
#pragma unroll
    for (int u = 0; u < CH; ++u) {
        const bool in = q + u < s1;
        jj[u] = in ? bcol[q + u] : -1;
        pp[u] = in ? __ldcg(prod + (q + u - s0)) : 0.0f;
    }
    bool more = true;
#pragma unroll
    for (int u = 0; u < CH; ++u) {
        more = more && jj[u] == j;
        if (more) delta = __fadd_rn(delta, pp[u]);
    }
    q += CH;
    return more;
}

// Runs longer than this many terms are summed by a whole warp.
constexpr int BSP_LONG = 16;

// Feature j's run from q, summed by the whole warp: 32 terms per load, the
// adds in ascending order on every lane (each lane ends with the same delta).
__device__ __forceinline__ float warp_run_sum(int32_t j, int64_t q, int64_t s0, int64_t s1,
                                              const int32_t *__restrict__ bcol, const float *prod)
{
    const int lane = threadIdx.x & 31;
    float delta = 0.0f;
    int32_t jn = q + lane < s1 ? bcol[q + lane] : -1;
    float pn = q + lane < s1 ? __ldcg(prod + (q + lane - s0)) : 0.0f;
    for (;;) {
        const float pc = pn;
        const int n = __popc(__ballot_sync(FULL, jn == j));   // the run is a prefix of the 32
        if (n == 32) {                                          // next 32 in flight during the adds
            q += 32;
            jn = q + lane < s1 ? bcol[q + lane] : -1;
            pn = q + lane < s1 ? __ldcg(prod + (q + lane - s0)) : 0.0f;
        }
#pragma unroll
        for (int u = 0; u < 32; ++u) {
            const float v = __shfl_sync(FULL, pc, u);
            if (u < n) delta = __fadd_rn(delta, v);
        }
        if (n < 32) return delta;
    }
}

// Algorithm 2a with B examples per step: reads (the margins at the batch-start
// weights), barrier; the products c_i * x_ij of the batch's pairs, which are
// pre-sorted by (batch, feature, example), barrier; writes (each feature's
// products summed in ascending example order, one run of the sorted pairs),
// barrier.  A feature's run is summed by one thread, or by a whole warp when
// it is longer than BSP_LONG terms.  Batches without such runs (has_long[b] =
// 0) skip the products step: each thread forms its run's products itself.
__global__ __launch_bounds__(THREADS, 8) void k_bsp(int32_t n_rows, int64_t batch, int64_t n_batches,
                                                 const int64_t *__restrict__ row_ptr, const int32_t *__restrict__ col,
                                                 const float *__restrict__ val, const float *__restrict__ y,
                                                 const int64_t *__restrict__ bptr, const int32_t *__restrict__ bcol,
                                                 const int32_t *__restrict__ brow, const float *__restrict__ bval,
                                                 const uint8_t *__restrict__ has_long, float *cbuf, float *prod,
                                                 float *w, int loss, float eta, int epochs,
                                                 GridBarrier *bar, int *status, uint64_t timeout)
{
    if (read_status(status)) return;
    const int lane = threadIdx.x & 31;
    const int64_t gtid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t nthr = (int64_t)gridDim.x * blockDim.x;
    const int gw = (int)(gtid >> 5), nw = (int)(nthr >> 5);
    for (int ep = 0; ep < epochs; ++ep)
        for (int64_t bi = 0; bi < n_batches; ++bi) {
            const int64_t r0 = bi * batch, r1 = min64(n_rows, r0 + batch);
            for (int64_t t = r0 + gw; t < r1; t += nw) {
                float m = margin((int)t, row_ptr, col, val, w);
                if (lane == 0) cbuf[t - r0] = __fmul_rn(eta, dev_grad(loss, m, y[t]));
            }
            if (!grid_sync(bar, status, timeout)) return;
            const int64_t s0 = bptr[bi], s1 = bptr[bi + 1];
            if (!has_long[bi]) {
                // every run is short: one thread per run, term by term
                for (int64_t s = s0 + gtid; s < s1; s += nthr) {
                    const int32_t j = bcol[s];
                    if (s > s0 && bcol[s - 1] == j) continue;
                    float delta = 0.0f;
                    for (int64_t q = s; q < s1 && bcol[q] == j; ++q) {
                        const int64_t i = brow[q] - r0;
                        if (i < 0 || i >= r1 - r0) {     // cannot happen with a consistent batch sort
                            set_status(status, PDB_EFAULT);
                            break;
                        }
                        delta = __fadd_rn(delta, __fmul_rn(__ldcg(cbuf + i), bval[q]));
                    }
                    __stcg(w + j, __fsub_rn(__ldcg(w + j), delta));
                }
                if (!grid_sync(bar, status, timeout)) return;
                continue;
            }
            for (int64_t s = s0 + gtid; s < s1; s += nthr) {
                int64_t i = brow[s] - r0;
                if (i < 0 || i >= r1 - r0) {     // cannot happen with a consistent batch sort
                    set_status(status, PDB_EFAULT);
                    i = 0;
                }
                __stcg(prod + (s - s0), __fmul_rn(__ldcg(cbuf + i), bval[s]));
            }
            if (!grid_sync(bar, status, timeout)) return;
            for (int64_t base = s0 + (int64_t)gw * 32; base < s1; base += (int64_t)nw * 32) {
                const int64_t s = base + lane;
                const int32_t j = s < s1 ? bcol[s] : -1;
                const bool start = s < s1 && (s == s0 || bcol[s - 1] != j);
                const bool is_long = start && s + BSP_LONG < s1 && bcol[s + BSP_LONG] == j;
                if (start && !is_long) {
                    // at most BSP_LONG terms: a short first chunk (most runs hold one or two)
                    float delta = 0.0f;
                    int64_t q = s;
                    if (run_chunk_prod<2>(j, q, s0, s1, bcol, prod, delta) &&
                        run_chunk_prod<8>(j, q, s0, s1, bcol, prod, delta))
                        run_chunk_prod<8>(j, q, s0, s1, bcol, prod, delta);
                    __stcg(w + j, __fsub_rn(__ldcg(w + j), delta));
                }
                for (unsigned lm = __ballot_sync(FULL, is_long); lm; lm &= lm - 1) {
                    const int src = __ffs(lm) - 1;
                    const int64_t sr = __shfl_sync(FULL, s, src);
                    const int32_t jr = __shfl_sync(FULL, j, src);
                    const float delta = warp_run_sum(jr, sr, s0, s1, bcol, prod);
                    if (lane == 0) __stcg(w + jr, __fsub_rn(__ldcg(w + jr), delta));
                }
            }
            if (!grid_sync(bar, status, timeout)) return;
        }
}

// has_long[b] = 1 when batch b holds a feature run longer than BSP_LONG terms
// (skey: batch of each pair in the (batch, feature, example) order)
__global__ void k_bsp_long(const uint32_t *__restrict__ skey, const int32_t *__restrict__ bcol, int64_t nnz,
                           uint8_t *__restrict__ has_long, const int *status)
{
    if (read_status(status)) return;
    for (int64_t s = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; s + BSP_LONG < nnz;
         s += (int64_t)gridDim.x * blockDim.x)
        if (bcol[s + BSP_LONG] == bcol[s] && skey[s + BSP_LONG] == skey[s]) has_long[skey[s]] = 1;
}

__global__ void k_bsp_keys(const int32_t *__restrict__ csc_pos, const int32_t *__restrict__ row_of, int64_t nnz,
                           int64_t batch, uint32_t *__restrict__ key, const int *status)
{
    if (read_status(status)) return;
    for (int64_t s = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; s < nnz; s += (int64_t)gridDim.x * blockDim.x)
        key[s] = (uint32_t)(row_of[csc_pos[s]] / batch);
}

__global__ void k_bsp_gather(const int32_t *__restrict__ bpos, const int32_t *__restrict__ col,
                             const float *__restrict__ val, const int32_t *__restrict__ row_of, int64_t nnz,
                             int32_t *__restrict__ bcol, int32_t *__restrict__ brow, float *__restrict__ bval,
                             const int *status)
{
    if (read_status(status)) return;
    for (int64_t s = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; s < nnz; s += (int64_t)gridDim.x * blockDim.x) {
        int32_t p = bpos[s];
        bcol[s] = col[p];
        brow[s] = row_of[p];
        bval[s] = val ? val[p] : 1.0f;
    }
}

// ---- Algorithm 2a split over data-parallel ranks (pdb_bsp_plan / coef / apply)
// c_i = eta * dloss/dm(m_i(w), y_i) for the rows [r0, r1), one warp per example,
// w the weights of the batch start (the read half of the step)
__global__ void k_bsp_coef(int64_t r0, int64_t r1, const int64_t *__restrict__ row_ptr,
                           const int32_t *__restrict__ col, const float *__restrict__ val,
                           const float *__restrict__ y, const float *w, int loss, float eta, float *__restrict__ coef,
                           const int *status)
{
    if (read_status(status)) return;
    const int lane = threadIdx.x & 31;
    const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t t = r0 + gw; t < r1; t += nw) {
        const float m = margin((int)t, row_ptr, col, val, w);
        if (lane == 0) coef[t - r0] = __fmul_rn(eta, dev_grad(loss, m, y[t]));
    }
}

// The write half of one batch: each feature's terms c_i * x_ij summed in
// ascending example order from +0, then w_j = w_j - delta_j.  The batch's
// pairs [s0, s1) are sorted by (feature, example); coef holds the whole
// batch's coefficients (rows r0.. in order).  A run of at most BSP_LONG
// terms is summed by one thread; a longer one by a whole warp, 32 terms per
// load with the same adds in the same order on every lane.
__global__ void k_bsp_apply(int64_t s0, int64_t s1, int64_t r0, int64_t rows, const int32_t *__restrict__ bcol,
                            const int32_t *__restrict__ brow, const float *__restrict__ bval,
                            const float *__restrict__ coef, float *w, int *status)
{
    if (read_status(status)) return;
    const int lane = threadIdx.x & 31;
    const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    bool bad = false;
    for (int64_t base = s0 + gw * 32; base < s1; base += nw * 32) {
        const int64_t s = base + lane;
        const int32_t j = s < s1 ? bcol[s] : -1;
        const bool start = s < s1 && (s == s0 || bcol[s - 1] != j);
        const bool is_long = start && s + BSP_LONG < s1 && bcol[s + BSP_LONG] == j;
        if (start && !is_long) {
            float delta = 0.0f;
            for (int64_t q = s; q < s1 && bcol[q] == j; ++q) {
                const int64_t i = brow[q] - r0;
                bad |= i < 0 || i >= rows;
                if (i >= 0 && i < rows) delta = __fadd_rn(delta, __fmul_rn(coef[i], bval[q]));
            }
            w[j] = __fsub_rn(w[j], delta);
        }
        for (unsigned lm = __ballot_sync(FULL, is_long); lm; lm &= lm - 1) {
            const int src = __ffs(lm) - 1;
            int64_t q = __shfl_sync(FULL, s, src);
            const int32_t jr = __shfl_sync(FULL, j, src);
            float delta = 0.0f;
            for (;;) {
                const bool in = q + lane < s1 && bcol[q + lane] == jr;
                float pv = 0.0f;
                if (in) {
                    const int64_t i = brow[q + lane] - r0;
                    bad |= i < 0 || i >= rows;
                    if (i >= 0 && i < rows) pv = __fmul_rn(coef[i], bval[q + lane]);
                }
                const int n = __popc(__ballot_sync(FULL, in));   // the run is a prefix of the 32
#pragma unroll
                for (int u = 0; u < 32; ++u) {
                    const float v = __shfl_sync(FULL, pv, u);
                    if (u < n) delta = __fadd_rn(delta, v);
                }
                if (n < 32) break;
                q += 32;
            }
            if (lane == 0) w[jr] = __fsub_rn(w[jr], delta);
        }
    }
    if (__any_sync(FULL, bad) && lane == 0) set_status(status, PDB_EFAULT);   // cannot happen with a consistent plan
}

__global__ void k_eval_grad(const float *__restrict__ m, const float *__restrict__ y, float *__restrict__ out,
                            int64_t n, int loss)
{
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        out[i] = dev_grad(loss, m[i], y[i]);
}

__global__ void k_eval_expf(const float *__restrict__ x, float *__restrict__ out, int64_t n)
{
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        out[i] = dev_expf(x[i]);
}

// Registers per lane for the example's elements: the smallest of 2, 4, 8
// that holds the longest row in registers (longer rows take the two-pass
// path).  The longest row is recorded by the conflict build; this waits for
// that build to finish if it has not.
int register_width(const pdb_conflicts *c)
{
    if (cudaEventSynchronize(c->ev1) != cudaSuccess) {
        cudaGetLastError();
        return 8;
    }
    const int longest = c->h_info[2];
    return longest <= 64 ? 2 : longest <= 128 ? 4 : 8;
}

int check_run(const pdb_csr *X, const float *y, const pdb_conflicts *c, const float *w, int loss, int epochs)
{
    if (!X || !c || epochs < 0) return PDB_EINVAL;
    if (loss != PDB_LOSS_LOGISTIC && loss != PDB_LOSS_SQUARED && loss != PDB_LOSS_HINGE) return PDB_EINVAL;
    if (X->n_rows != c->n_rows || X->n_cols != c->n_cols || X->nnz != c->nnz) return PDB_EINVAL;
    if (!X->row_ptr || (X->nnz > 0 && !X->col)) return PDB_EINVAL;
    if ((X->n_rows > 0 && !y) || (X->n_cols > 0 && !w)) return PDB_EINVAL;
    return PDB_OK;
}

}  // namespace

extern "C" {

int pdb_sgd_epoch(const pdb_csr *X, const float *y, const pdb_conflicts *c, const pdb_schedule *h, float *w,
                  pdb_loss loss, float eta, int n_epochs, const pdb_opts *opts, void *stream)
{
    ApiScope scope("pdb_sgd_epoch", c, h);
    UseMark use{c, h, (cudaStream_t)stream};
    int rc = check_run(X, y, c, w, loss, n_epochs);
    if (rc != PDB_OK) return rc;
    if (!h || h->c != c) return PDB_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    pdb_conflicts *cm = const_cast<pdb_conflicts *>(c);
    const int width = register_width(cm);
    cudaEventRecord(cm->ev_sgd0, s);
    cudaEventRecord(cm->ev_k0, s);
    cudaEventRecord(cm->ev_k1, s);
    const uint64_t tmo = timeout_ns(opts);
    uint64_t *trace = opts ? opts->trace : nullptr;
    int32_t n32 = (int32_t)X->n_rows;
    int lossi = (int)loss;
    if (X->n_rows > 0 && n_epochs > 0) {
        if (h->mode == PDB_SCHED_LEVELS) {
            const void *kern = width == 2 ? (const void *)k_sgd_levels<2>
                               : width == 4 ? (const void *)k_sgd_levels<4> : (const void *)k_sgd_levels<8>;
            int grid = persistent_grid(kern, opts);
            const int64_t *rp = X->row_ptr;
            const int32_t *cl = X->col;
            const float *vl = X->val;
            void *args[] = {(void *)&n32,      (void *)&rp,  (void *)&cl,       (void *)&vl,     (void *)&y,
                            (void *)&h->order, (void *)&h->level_ptr, (void *)&h->ctl, (void *)&w,
                            (void *)&lossi,    (void *)&eta, (void *)&n_epochs, (void *)&h->bar,
                            (void *)&cm->status, (void *)&tmo, (void *)&trace};
            cudaEventRecord(cm->ev_k0, s);
            if (cudaLaunchCooperativeKernel(kern, grid, THREADS, args, 0, s) != cudaSuccess) rc = PDB_ECUDA;
            note_launch();
            cudaEventRecord(cm->ev_k1, s);
        } else if (h->mode == PDB_SCHED_CHAIN) {
            cudaEventRecord(cm->ev_k0, s);
            rc = h->resident ? resident_run(X, y, w, lossi, eta, n_epochs, c->h_info[2], cm->status, trace, s)
                             : chain_run(X, y, h->link, w, lossi, eta, n_epochs, c->h_info[2], cm->status, trace, s);
            cudaEventRecord(cm->ev_k1, s);
        } else if (h->mode == PDB_SCHED_WINDOW) {
            cudaEventRecord(cm->ev_k0, s);
            pdb_schedule *hm = const_cast<pdb_schedule *>(h);
            rc = window_run(X, y, c->gate_window, w, h->rec, &hm->epochs_run, h->prog, h->prog_cap, h->wctl, c->near, lossi,
                            eta, n_epochs, width, opts, cm->status, tmo, s);
            cudaEventRecord(cm->ev_k1, s);
        } else if (block_ready_smem(X->n_cols, c->h_info[2]) > 0 && (int64_t)n_epochs * X->n_rows < (1ll << 31)) {
            // READY with every record in one block's shared memory (few features)
            cudaEventRecord(cm->ev_k0, s);
            rc = block_ready_run(X, y, c->gate, w, lossi, eta, n_epochs, c->h_info[2], cm->status, tmo, trace, s);
            cudaEventRecord(cm->ev_k1, s);
        } else {
            auto kern = width == 2 ? k_sgd_ready<2> : width == 4 ? k_sgd_ready<4> : k_sgd_ready<8>;
            int grid = persistent_grid((const void *)kern, opts);
            const int64_t F = X->n_cols;
            const int chunk = (opts && opts->ticket_chunk > 0) ? opts->ticket_chunk : 2;
            k_pack<<<grid_1d(F), 256, 0, s>>>(w, F, h->rec, cm->status);
            note_launch();
            if (fill_words(h->ticket, 0u, sizeof(unsigned long long), s) != PDB_OK) return PDB_ECUDA;
            cudaEventRecord(cm->ev_k0, s);
            kern<<<grid, THREADS, 0, s>>>(n32, X->row_ptr, X->col, X->val, y, c->gate, h->rec, lossi, eta, n_epochs,
                                          h->ticket, chunk, cm->status, tmo, trace);
            note_launch();
            cudaEventRecord(cm->ev_k1, s);
            k_unpack<<<grid_1d(F), 256, 0, s>>>(h->rec, F, w, cm->status);
            note_launch();
        }
    }
    cudaEventRecord(cm->ev_sgd1, s);
    cm->timed_sgd = true;
    if (rc == PDB_OK && cudaPeekAtLastError() != cudaSuccess) rc = PDB_ECUDA;
    if (rc != PDB_OK) cudaGetLastError();
    return rc;
}

int pdb_ssp_epoch(const pdb_csr *X, const float *y, const pdb_conflicts *c, const pdb_schedule *h, float *w,
                  pdb_loss loss, float eta, int n_epochs, int64_t delay, float *coef, const pdb_opts *opts,
                  void *stream)
{
    ApiScope scope("pdb_ssp_epoch", c, h);
    UseMark use{c, h, (cudaStream_t)stream};
    int rc = check_run(X, y, c, w, loss, n_epochs);
    if (rc != PDB_OK) return rc;
    if (!h || h->c != c || delay < 0) return PDB_EINVAL;
    if (h->mode != PDB_SCHED_READY) return PDB_ESTATE;
    const int gates = opts ? opts->ssp_gates : 0;
    if (gates < 0 || gates > PDB_SSP_PREFIX) return PDB_EINVAL;
    const bool prefix = gates == PDB_SSP_PREFIX;
    cudaStream_t s = (cudaStream_t)stream;
    pdb_conflicts *cm = const_cast<pdb_conflicts *>(c);
    pdb_schedule *hm = const_cast<pdb_schedule *>(h);
    const int width = register_width(cm);
    // scratch kept with the schedule, allocated in pairs on first use and
    // attached only when both allocations succeeded
    auto alloc_pair = [&](unsigned **a, unsigned **b, int64_t words) {
        if (*a && *b) return PDB_OK;
        unsigned *x = nullptr, *z = nullptr;
        int r = alloc((void **)&x, sizeof(unsigned) * words, s);
        r = r ? r : alloc((void **)&z, sizeof(unsigned) * words, s);
        if (r != PDB_OK) {
            release(x, s);
            release(z, s);
            return r;
        }
        release(*a, s);
        release(*b, s);
        *a = x;
        *b = z;
        return PDB_OK;
    };
    rc = alloc_pair(&hm->reads, &hm->writes, std::max<int64_t>(X->n_cols, 1));
    if (rc != PDB_OK) return rc;
    // one bit per CSC slot, two words of slack past the last slot's word
    const int64_t n_words = X->nnz / 32 + 2;
    if (prefix) {
        rc = alloc_pair(&hm->rbits, &hm->wbits, n_words);
        if (rc != PDB_OK) return rc;
    }
    cudaEventRecord(cm->ev_sgd0, s);
    cudaEventRecord(cm->ev_k0, s);
    if (X->n_rows > 0 && n_epochs > 0)
        rc = ssp_run(X, y, c->gate, w, hm->writes, hm->reads, h->ticket, (long long)std::min<int64_t>(delay, 1ll << 40),
                     coef, (int)loss, eta, n_epochs, width, opts, cm->status, timeout_ns(opts), s, c->feat_ptr,
                     prefix ? hm->rbits : nullptr, prefix ? hm->wbits : nullptr, n_words);
    cudaEventRecord(cm->ev_k1, s);
    cudaEventRecord(cm->ev_sgd1, s);
    cm->timed_sgd = true;
    if (rc == PDB_OK && cudaPeekAtLastError() != cudaSuccess) rc = PDB_ECUDA;
    if (rc != PDB_OK) cudaGetLastError();
    return rc;
}

int pdb_bsp_epoch(const pdb_csr *X, const float *y, const pdb_conflicts *c, float *w, pdb_loss loss, float eta,
                  int64_t batch, int n_epochs, const pdb_opts *opts, void *stream)
{
    ApiScope scope("pdb_bsp_epoch", c);
    UseMark use{c, nullptr, (cudaStream_t)stream};
    int rc = check_run(X, y, c, w, loss, n_epochs);
    if (rc != PDB_OK) return rc;
    if (batch < 1) return PDB_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    pdb_conflicts *cm = const_cast<pdb_conflicts *>(c);
    const int64_t N = X->n_rows, nnz = X->nnz;
    if (batch > N && N > 0) batch = N;
    cudaEventRecord(cm->ev_bsp0, s);
    if (N > 0 && n_epochs > 0) {
        const int64_t n_batches = (N + batch - 1) / batch;
        uint32_t *key = nullptr, *skey = nullptr, *tkey = nullptr;
        int32_t *bpos = nullptr, *tval = nullptr, *bcol = nullptr, *brow = nullptr;
        float *bval = nullptr, *cbuf = nullptr, *prod = nullptr;
        uint8_t *has_long = nullptr;
        int64_t *bptr = nullptr;
        GridBarrier *bar = nullptr;
        rc = alloc((void **)&key, sizeof(uint32_t) * nnz, s);
        rc = rc ? rc : alloc((void **)&skey, sizeof(uint32_t) * nnz, s);
        rc = rc ? rc : alloc((void **)&tkey, sizeof(uint32_t) * nnz, s);
        rc = rc ? rc : alloc((void **)&bpos, sizeof(int32_t) * nnz, s);
        rc = rc ? rc : alloc((void **)&tval, sizeof(int32_t) * nnz, s);
        rc = rc ? rc : alloc((void **)&bcol, sizeof(int32_t) * nnz, s);
        rc = rc ? rc : alloc((void **)&brow, sizeof(int32_t) * nnz, s);
        rc = rc ? rc : alloc((void **)&bval, sizeof(float) * nnz, s);
        rc = rc ? rc : alloc((void **)&cbuf, sizeof(float) * batch, s);
        // products of the largest batch: at most batch x (longest row) pairs
        int64_t max_row = 0;
        if (rc == PDB_OK) {
            if (cudaEventSynchronize(c->ev1) != cudaSuccess) {
                cudaGetLastError();
                rc = PDB_ECUDA;
            }
            max_row = c->h_info[2];
        }
        rc = rc ? rc : alloc((void **)&has_long, (size_t)n_batches, s);
        rc = rc ? rc : alloc((void **)&prod, sizeof(float) * std::max<int64_t>(1, std::min<int64_t>(nnz, batch * max_row)), s);
        rc = rc ? rc : alloc((void **)&bptr, sizeof(int64_t) * (n_batches + 1), s);
        rc = rc ? rc : alloc((void **)&bar, sizeof(GridBarrier), s);
        if (rc == PDB_OK) {
            rc = fill_words(bar, 0u, sizeof(GridBarrier), s);
            if (rc == PDB_OK && nnz > 0) rc = ensure_row_of(cm, s);
            if (rc == PDB_OK && nnz > 0) {
                k_bsp_keys<<<grid_1d(nnz), 256, 0, s>>>(c->csc_pos, c->row_of, nnz, batch, key, cm->status); note_launch();
                // stable by batch: inside a batch the feature-major CSC order survives
                rc = radix_sort(key, c->csc_pos, skey, bpos, tkey, tval, nnz, bits_for(n_batches - 1), cm->status, s);
                if (rc == PDB_OK)
                    k_bsp_gather<<<grid_1d(nnz), 256, 0, s>>>(bpos, X->col, X->val, c->row_of, nnz, bcol, brow, bval,
                                                              cm->status); note_launch();
            }
            if (rc == PDB_OK) rc = segment_bounds(skey, nnz, n_batches, nullptr, bptr, cm->status, s);
            if (rc == PDB_OK) {
                cudaMemsetAsync(has_long, 0, (size_t)n_batches, s);
                if (nnz > BSP_LONG) {
                    k_bsp_long<<<grid_1d(nnz), 256, 0, s>>>(skey, bcol, nnz, has_long, cm->status);
                    note_launch();
                }
            }
            if (rc == PDB_OK) {
                const void *kern = (const void *)k_bsp;
                int grid = persistent_grid(kern, opts);
                int32_t n32 = (int32_t)N;
                int lossi = (int)loss;
                uint64_t tmo = timeout_ns(opts);
                const int64_t *rp = X->row_ptr;
                const int32_t *cl = X->col;
                const float *vl = X->val;
                void *args[] = {&n32,  &batch, (void *)&n_batches, (void *)&rp, (void *)&cl, (void *)&vl,
                                (void *)&y, &bptr, &bcol, &brow, &bval, &has_long, &cbuf, &prod, &w, &lossi, &eta, &n_epochs, &bar,
                                (void *)&cm->status, &tmo};
                if (cudaLaunchCooperativeKernel(kern, grid, THREADS, args, 0, s) != cudaSuccess) rc = PDB_ECUDA; note_launch();
            }
        }
        for (void *p : {(void *)key, (void *)skey, (void *)tkey, (void *)bpos, (void *)tval, (void *)bcol, (void *)brow,
                        (void *)bval, (void *)cbuf, (void *)prod, (void *)has_long, (void *)bptr, (void *)bar})
            release(p, s);
    }
    cudaEventRecord(cm->ev_bsp1, s);
    cm->timed_bsp = true;
    if (rc == PDB_OK && cudaPeekAtLastError() != cudaSuccess) rc = PDB_ECUDA;
    if (rc != PDB_OK) cudaGetLastError();
    return rc;
}

int pdb_bsp_plan_build(const pdb_conflicts *c, int64_t batch, pdb_bsp_plan **out, void *stream)
{
    ApiScope scope("pdb_bsp_plan_build", c);
    if (!out) return PDB_EINVAL;
    *out = nullptr;
    if (!c || batch < 1) return PDB_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    pdb_conflicts *cm = const_cast<pdb_conflicts *>(c);
    const int64_t N = c->n_rows, nnz = c->nnz;
    if (batch > N && N > 0) batch = N;
    pdb_bsp_plan *p = new (std::nothrow) pdb_bsp_plan();
    if (!p) return PDB_ENOMEM;
    p->c = c;
    p->batch = batch;
    if (cudaEventCreateWithFlags(&p->ev_use, cudaEventDisableTiming) != cudaSuccess) {
        cudaGetLastError();
        p->ev_use = nullptr;
    }
    p->n_batches = N > 0 ? (N + batch - 1) / batch : 0;
    uint32_t *key = nullptr, *skey = nullptr, *tkey = nullptr;
    int32_t *bpos = nullptr, *tval = nullptr;
    int rc = alloc((void **)&p->bptr, sizeof(int64_t) * (p->n_batches + 1), s);
    if (rc == PDB_OK && nnz > 0) {
        rc = alloc((void **)&p->bcol, sizeof(int32_t) * nnz, s);
        rc = rc ? rc : alloc((void **)&p->brow, sizeof(int32_t) * nnz, s);
        rc = rc ? rc : alloc((void **)&p->bval, sizeof(float) * nnz, s);
        rc = rc ? rc : alloc((void **)&key, sizeof(uint32_t) * nnz, s);
        rc = rc ? rc : alloc((void **)&skey, sizeof(uint32_t) * nnz, s);
        rc = rc ? rc : alloc((void **)&tkey, sizeof(uint32_t) * nnz, s);
        rc = rc ? rc : alloc((void **)&bpos, sizeof(int32_t) * nnz, s);
        rc = rc ? rc : alloc((void **)&tval, sizeof(int32_t) * nnz, s);
        rc = rc ? rc : ensure_row_of(cm, s);
        if (rc == PDB_OK) {
            k_bsp_keys<<<grid_1d(nnz), 256, 0, s>>>(c->csc_pos, c->row_of, nnz, batch, key, cm->status);
            note_launch();
            // stable by batch: inside a batch the feature-major CSC order survives
            rc = radix_sort(key, c->csc_pos, skey, bpos, tkey, tval, nnz, bits_for(p->n_batches - 1), cm->status, s);
        }
        if (rc == PDB_OK) {
            k_bsp_gather<<<grid_1d(nnz), 256, 0, s>>>(bpos, c->col, c->val, c->row_of, nnz, p->bcol, p->brow, p->bval,
                                                      cm->status);
            note_launch();
            rc = segment_bounds(skey, nnz, p->n_batches, nullptr, p->bptr, cm->status, s);
        }
    } else if (rc == PDB_OK) {
        rc = fill_words(p->bptr, 0u, sizeof(int64_t) * (p->n_batches + 1), s);
    }
    for (void *q : {(void *)key, (void *)skey, (void *)tkey, (void *)bpos, (void *)tval}) release(q, s);
    if (rc == PDB_OK && cudaPeekAtLastError() != cudaSuccess) rc = PDB_ECUDA;
    // the host keeps the batches' pair bounds (apply needs them to size its launch)
    if (rc == PDB_OK) {
        p->h_bptr = new (std::nothrow) int64_t[p->n_batches + 1];
        if (!p->h_bptr) rc = PDB_ENOMEM;
        else if (cudaMemcpyAsync(p->h_bptr, p->bptr, sizeof(int64_t) * (p->n_batches + 1), cudaMemcpyDeviceToHost, s) !=
                     cudaSuccess ||
                 cudaStreamSynchronize(s) != cudaSuccess)
            rc = PDB_ECUDA;
    }
    if (rc != PDB_OK) {
        cudaGetLastError();
        cudaStreamSynchronize(s);
        pdb_bsp_plan_free(p);
        return rc;
    }
    *out = p;
    return PDB_OK;
}

int64_t pdb_bsp_plan_batches(const pdb_bsp_plan *p) { return p ? p->n_batches : -1; }

int pdb_bsp_coef(const pdb_bsp_plan *p, const pdb_csr *X, const float *y, const float *w, pdb_loss loss, float eta,
                 int64_t row_begin, int64_t row_end, float *coef, void *stream)
{
    ApiScope scope("pdb_bsp_coef", p ? p->c : nullptr, nullptr, nullptr, nullptr, false);
    UseMark use{p ? p->c : nullptr, nullptr, (cudaStream_t)stream};
    if (!p) return PDB_EINVAL;
    int rc = check_run(X, y, p->c, w, loss, 1);
    if (rc != PDB_OK) return rc;
    if (row_begin < 0 || row_end < row_begin || row_end > X->n_rows) return PDB_EINVAL;
    if (row_end > row_begin && !coef) return PDB_EINVAL;
    // the rows must lie inside one batch: the margins read that batch's start weights
    if (row_end > row_begin && row_begin / p->batch != (row_end - 1) / p->batch) return PDB_EINVAL;
    if (row_end == row_begin) return PDB_OK;
    cudaStream_t s = (cudaStream_t)stream;
    k_bsp_coef<<<grid_1d((row_end - row_begin) * 32), 256, 0, s>>>(row_begin, row_end, X->row_ptr, X->col, X->val, y,
                                                                  w, (int)loss, eta, coef, p->c->status);
    note_launch();
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

int pdb_bsp_apply(const pdb_bsp_plan *p, float *w, int64_t batch_index, const float *coef, void *stream)
{
    ApiScope scope("pdb_bsp_apply", p ? p->c : nullptr, nullptr, nullptr, nullptr, false);
    UseMark use{p ? p->c : nullptr, nullptr, (cudaStream_t)stream};
    if (!p || batch_index < 0 || batch_index >= p->n_batches) return PDB_EINVAL;
    if (p->c->n_cols > 0 && !w) return PDB_EINVAL;
    const int64_t s0 = p->h_bptr[batch_index], s1 = p->h_bptr[batch_index + 1];
    if (s1 == s0) return PDB_OK;
    if (!coef) return PDB_EINVAL;
    const int64_t r0 = batch_index * p->batch, rows = std::min(p->c->n_rows, r0 + p->batch) - r0;
    cudaStream_t s = (cudaStream_t)stream;
    const int64_t blocks = std::max<int64_t>(1, std::min<int64_t>((s1 - s0 + 255) / 256, (int64_t)152 * 16));
    k_bsp_apply<<<(unsigned)blocks, 256, 0, s>>>(s0, s1, r0, rows, p->bcol, p->brow, p->bval, coef, w,
                                                 const_cast<pdb_conflicts *>(p->c)->status);
    note_launch();
    if (p->ev_use) cudaEventRecord(p->ev_use, s);
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

void pdb_bsp_plan_free(pdb_bsp_plan *p)
{
    if (!p) return;
    // the plan's own work only: other streams of the device keep running
    if (p->ev_use) {
        cudaEventSynchronize(p->ev_use);
        cudaEventDestroy(p->ev_use);
    }
    cudaGetLastError();
    for (void *q : {(void *)p->bptr, (void *)p->bcol, (void *)p->brow, (void *)p->bval})
        if (q) cudaFreeAsync(q, own_stream());
    delete[] p->h_bptr;
    delete p;
}

int pdb_eval_grad(const float *m, const float *y, float *out, int64_t n, pdb_loss loss, void *stream)
{
    if (n < 0 || (n > 0 && (!m || !y || !out))) return PDB_EINVAL;
    if (loss != PDB_LOSS_LOGISTIC && loss != PDB_LOSS_SQUARED && loss != PDB_LOSS_HINGE) return PDB_EINVAL;
    if (n == 0) return PDB_OK;
    k_eval_grad<<<grid_1d(n), 256, 0, (cudaStream_t)stream>>>(m, y, out, n, (int)loss);
    note_launch();
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

int pdb_eval_expf(const float *x, float *out, int64_t n, void *stream)
{
    if (n < 0 || (n > 0 && (!x || !out))) return PDB_EINVAL;
    if (n == 0) return PDB_OK;
    k_eval_expf<<<grid_1d(n), 256, 0, (cudaStream_t)stream>>>(x, out, n); note_launch();
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

}  // extern "C"

// ---------------------------------------------------------------- allocation-free READY epoch
// Some callers cannot let a library allocate device memory while they
// train: a server that has handed all device memory to its own pool and
// must not see it grow or fragment, or a host runtime that accounts for
// every device allocation itself and forbids libraries to make their own.
// For them the READY epoch below keeps its per-feature (weight, version)
// records, its ticket counter and its status word in one fixed array
// compiled into the library instead of in a schedule handle.  Every GPU that
// loads libpdb holds this array (NOALLOC_MAX_COLS * 8 bytes + 256 bytes,
// about 8 MiB) until the process exits.  All calls on a device share it:
// two calls whose work overlaps on the GPU corrupt each other, so order them
// on one stream.
constexpr int64_t NOALLOC_MAX_COLS = 1 << 20;
constexpr int64_t NOALLOC_WORDS = NOALLOC_MAX_COLS + 32;   // records, then ticket and status
static __device__ __align__(256) unsigned long long g_noalloc_scratch[NOALLOC_WORDS];

namespace {

std::mutex g_noalloc_lock;
struct NoallocSlot {
    void *ctx;                  // context the address was looked up in
    unsigned long long *ptr;
};
NoallocSlot g_noalloc_slot[64];

// The driver's current context (nullptr when none is current or the driver
// entry point is unavailable).  A device's module, and with it the scratch
// array, is loaded once per context: after cudaDeviceReset the array may sit
// elsewhere, so the cached address is keyed by context as well as device.
void *current_context()
{
    typedef CUresult (*GetCurrent)(CUcontext *);
    static GetCurrent fn = [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess) {
            cudaGetLastError();
            return (GetCurrent) nullptr;
        }
        return (GetCurrent)f;
    }();
    CUcontext c = nullptr;
    if (!fn || fn(&c) != CUDA_SUCCESS) return nullptr;
    return (void *)c;
}

// Device address of the scratch array for the current device and context.
// Host code only sees a stand-in symbol, not the address, so the address is
// looked up (cudaGetSymbolAddress, with that device current) on the first
// call in each device context and reused afterwards.
unsigned long long *noalloc_scratch()
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    std::lock_guard<std::mutex> guard(g_noalloc_lock);
    NoallocSlot &slot = g_noalloc_slot[dev];
    void *ctx = current_context();
    if (!slot.ptr || !ctx || ctx != slot.ctx) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) {
            cudaGetLastError();
            slot.ptr = nullptr;
            return nullptr;
        }
        slot.ptr = (unsigned long long *)p;
        slot.ctx = current_context();   // the lookup makes the device's primary context current
    }
    return slot.ptr;
}

}  // namespace

extern "C" int pdb_sgd_epoch_ready_noalloc(const pdb_csr *X, const float *y, const uint32_t *gate, float *w,
                                           pdb_loss loss, float eta, int n_epochs, void *stream)
{
    ApiScope scope("pdb_sgd_epoch_ready_noalloc", nullptr, nullptr, nullptr, nullptr, false);  // no handle to log
    if (!X || X->n_rows < 0 || X->n_cols < 0 || X->nnz < 0 || n_epochs < 0) return PDB_EINVAL;
    if (X->n_cols > NOALLOC_MAX_COLS) return PDB_ETOOBIG;
    if (X->n_rows >= (1ll << 31) - 1 || X->nnz >= (1ll << 31) - 1) return PDB_EINVAL;
    if (loss != PDB_LOSS_LOGISTIC && loss != PDB_LOSS_SQUARED && loss != PDB_LOSS_HINGE) return PDB_EINVAL;
    if (!X->row_ptr || (X->nnz > 0 && (!X->col || !gate)) || (X->n_rows > 0 && !y) || (X->n_cols > 0 && !w))
        return PDB_EINVAL;
    unsigned long long *scratch = noalloc_scratch();
    if (!scratch) return PDB_ECUDA;
    unsigned long long *rec = scratch;
    unsigned long long *ticket = scratch + NOALLOC_MAX_COLS;
    int *status = (int *)(scratch + NOALLOC_MAX_COLS + 1);
    cudaStream_t s = (cudaStream_t)stream;
    // the previous call left its status and ticket behind: start from zero
    if (fill_words(status, 0u, sizeof(int), s) != PDB_OK) return PDB_ECUDA;
    if (X->n_rows > 0 && n_epochs > 0) {
        const int64_t F = X->n_cols;
        const int32_t n32 = (int32_t)X->n_rows;
        const uint64_t tmo = timeout_ns(nullptr);
        const int grid = persistent_grid((const void *)k_sgd_ready<8>, nullptr);
        if (F > 0) {
            k_pack<<<grid_1d(F), 256, 0, s>>>(w, F, rec, status);
            note_launch();
        }
        if (fill_words(ticket, 0u, sizeof(unsigned long long), s) != PDB_OK) return PDB_ECUDA;
        k_sgd_ready<8><<<grid, THREADS, 0, s>>>(n32, X->row_ptr, X->col, X->val, y, gate, rec, (int)loss, eta,
                                                n_epochs, ticket, 2, status, tmo, nullptr);
        note_launch();
        if (F > 0) {
            k_unpack<<<grid_1d(F), 256, 0, s>>>(rec, F, w, status);
            note_launch();
        }
    }
    if (cudaPeekAtLastError() != cudaSuccess) {
        cudaGetLastError();
        return PDB_ECUDA;
    }
    int st = 0;
    if (cudaMemcpyAsync(&st, status, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
        return PDB_ECUDA;
    return st;
}
