// Admissible-delay engine: pdb_ssp_epoch (Section 7).
//
// The asynchronous Read and Write Constraints of Section 7, per feature as
// everywhere else in this library (an iteration = one example, a chunk = one
// feature, iteration numbers counted per feature):
//
//   read   the occurrence of feature j with rank r may read w_j once at least
//          r - delta writes of j are done (its view is at most delta
//          occurrences stale);
//   write  it may write once at least r - delta + 1 occurrences of j have
//          read, and it applies its step to the current w_j with an atomic
//          fp32 add of -(eta*g*x_j), then counts the write (release): no
//          update is lost even when a later occurrence wrote first, and
//          nothing retries.
//
// Counts equal the paper's per-iteration conditions only while reads and
// writes complete in rank order, which delta = 0 forces.  For delta >= 1 the
// read gate still bounds staleness from below, but the write gate counts any
// r - delta + 1 reads: a slow reader of low rank holds no writer back (the
// paper's Write Protocol waits for the slowest reader), so its read may see
// writes of occurrences delta or more ranks after it.
//
// delta = 0 is the sequential computation: the reader of rank r sees exactly
// r writes, nobody else writes between its read and its write, and
// w + (-(c*x)) rounds exactly as the sequential w - c*x, so the result is
// the READY engine's bit for bit.  delta > 0 admits more interleavings;
// results then depend on timing (not deterministic).  delta >= the longest
// chain is Hogwild with atomic updates (the paper's delta = infinity).
//
// Prefix gates (pdb_opts.ssp_gates = PDB_SSP_PREFIX), the paper's two
// protocols per feature: rank r reads once every rank <= r - 1 - delta has
// written, and writes once every rank <= r - delta has read (the Write
// Protocol's slowest reader).  A read then sees every write of rank
// <= r - 1 - delta and none of rank >= r + delta.  Per direction a done-bitmap
// over the CSC slots (rank r of j is slot feat_ptr[j] + r) is set by each
// occurrence after its access (red.release.or); the per-feature word that
// counts in the other form holds a prefix hint instead: ranks 0 .. hint-1 are
// known done.  A gate loads the hint; if it is short, it scans the bitmap
// from there for a run of set bits (clamped at what it needs), raises the
// hint to what it saw (red.release.max) and passes, or naps and scans again.
// No compare-and-swap loop, so a hot feature's word sees one reduction per
// occurrence, as under counting.
//
// Deadlock freedom: examples are taken in data order; the oldest unfinished
// example finds every earlier occurrence of its features read and written,
// so both of its waits pass, under either form.  Every wait is bounded by
// the timeout.
#include <cuda_runtime.h>

#include "common.cuh"

using namespace pdb;

namespace {

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned *p)
{
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void red_release_max(unsigned *p, unsigned v)
{
    asm volatile("red.release.gpu.global.max.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
// count one read or write of the feature, after the access it counts (release)
__device__ __forceinline__ void count_release(unsigned *p)
{
    asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(p) : "memory");
}

__device__ __forceinline__ bool keep_waiting(unsigned &spins, uint64_t t0, int *status, uint64_t timeout)
{
    if ((++spins & 15u) != 0) return true;
    if (read_status(status)) return false;
    if (globaltimer() - t0 > timeout) {
        set_status(status, PDB_ETIMEOUT);
        return false;
    }
    return true;
}

// waits until counter >= need (need <= 0: at once)
__device__ __forceinline__ bool wait_count(const unsigned *counter, long long need, int *status, uint64_t timeout)
{
    if (need <= 0 || (long long)ld_acquire_u32(counter) >= need) return true;
    const uint64_t t0 = globaltimer();
    unsigned spins = 0, nap = 32;
    for (;;) {
        __nanosleep(nap);
        nap = nap < 512 ? 2 * nap : 512;
        if ((long long)ld_acquire_u32(counter) >= need) return true;
        if (!keep_waiting(spins, t0, status, timeout)) return false;
    }
}

// w_j once at least `need` writes of j are done, then count the read
__device__ __forceinline__ bool read_admitted(const float *w, const unsigned *writes, unsigned *reads, int j,
                                              long long need, float &wv, int *status, uint64_t timeout)
{
    if (!wait_count(writes + j, need, status, timeout)) return false;
    wv = __ldcg(w + j);
    count_release(reads + j);
    return true;
}

// ranks 0 .. need-1 of a feature (slots fp + rank) are set in `bits`; hint
// caches a prefix known done.  Slots scanned stay below fp + need <= the
// feature's end, as need never exceeds its occurrence count.
__device__ __forceinline__ bool wait_prefix(const unsigned *bits, unsigned *hint, int64_t fp, long long need,
                                            int *status, uint64_t timeout)
{
    if (need <= 0) return true;
    long long p = ld_acquire_u32(hint);
    if (p >= need) return true;
    const uint64_t t0 = globaltimer();
    unsigned spins = 0, nap = 32;
    for (;;) {
        const long long start = p;
        for (;;) {
            const int64_t s = fp + p;
            const int b = (int)(s & 31);
            const unsigned x = ~(ld_acquire_u32(bits + (s >> 5)) >> b);   // zero where slot s + i is done
            const int t = x ? __ffs((int)x) - 1 : 32;                      // <= 32 - b: the top b bits of x are 1
            p = p + t < need ? p + t : need;
            if (p >= need || t < 32 - b) break;
        }
        if (p > start) red_release_max(hint, (unsigned)p);
        if (p >= need) return true;
        __nanosleep(nap);
        nap = nap < 512 ? 2 * nap : 512;
        if (!keep_waiting(spins, t0, status, timeout)) return false;
        const long long h = ld_acquire_u32(hint);
        if (h > p) p = h;
        if (p >= need) return true;   // before any scan: slots from fp + need on are not this wait's
    }
}

// mark slot s done (release: the access it stands for is visible first)
__device__ __forceinline__ void mark_release(unsigned *bits, int64_t s)
{
    asm volatile("red.release.gpu.global.or.b32 [%0], %1;" ::"l"(bits + (s >> 5)), "r"(1u << (s & 31)) : "memory");
}

// first slot of feature j; a rank at or past its occurrence count (a
// corrupted gate word) is PDB_EFAULT, so no bitmap access leaves the
// feature's slots
__device__ __forceinline__ bool slot_base(const int64_t *feat_ptr, int j, long long rank, int64_t &fp, int *status)
{
    fp = feat_ptr[j];
    if (rank >= 0 && rank < feat_ptr[j + 1] - fp) return true;
    set_status(status, PDB_EFAULT);
    return false;
}

// w_j once ranks 0 .. need-1 of j have written, then mark this read
__device__ __forceinline__ bool read_prefix(const float *w, const unsigned *wbits, unsigned *whint, unsigned *rbits,
                                            const int64_t *feat_ptr, int j, long long rank, long long need, float &wv,
                                            int *status, uint64_t timeout)
{
    int64_t fp;
    if (!slot_base(feat_ptr, j, rank, fp, status)) return false;
    if (!wait_prefix(wbits, whint + j, fp, need, status, timeout)) return false;
    wv = __ldcg(w + j);
    mark_release(rbits, fp + rank);
    return true;
}

// w_j -= step once ranks 0 .. need-1 of j have read, then mark this write
__device__ __forceinline__ bool write_prefix(float *w, unsigned *wbits, const unsigned *rbits, unsigned *rhint,
                                             const int64_t *feat_ptr, int j, long long rank, long long need, float step,
                                             int *status, uint64_t timeout)
{
    int64_t fp;
    if (!slot_base(feat_ptr, j, rank, fp, status)) return false;
    if (!wait_prefix(rbits, rhint + j, fp, need, status, timeout)) return false;
    atomicAdd(w + j, -step);
    mark_release(wbits, fp + rank);
    return true;
}

// w_j -= step once at least `need` reads of j are done, then count the write
__device__ __forceinline__ bool write_admitted(float *w, unsigned *writes, const unsigned *reads, int j,
                                               long long need, float step, int *status, uint64_t timeout)
{
    if (!wait_count(reads + j, need, status, timeout)) return false;
    atomicAdd(w + j, -step);
    count_release(writes + j);
    return true;
}

template <int R, bool PREFIX>
__global__ __launch_bounds__(THREADS) void k_sgd_ssp(int32_t n_rows, const int64_t *__restrict__ row_ptr,
                                                     const int32_t *__restrict__ col, const float *__restrict__ val,
                                                     const float *__restrict__ y, const uint32_t *__restrict__ gate,
                                                     float *w, unsigned *writes, unsigned *reads, long long delay,
                                                     float *coef, int loss, float eta, unsigned long long *ticket,
                                                     int chunk, int *status, uint64_t timeout, uint64_t *trace,
                                                     int64_t trace_base, const int64_t *__restrict__ feat_ptr,
                                                     unsigned *rbits, unsigned *wbits)
{
    if (read_status(status)) return;
    const int lane = threadIdx.x & 31;
    for (;;) {
        unsigned long long tk = 0;
        if (lane == 0) tk = atomicAdd(ticket, (unsigned long long)chunk);
        tk = __shfl_sync(FULL, tk, 0);
        if (tk >= (unsigned long long)n_rows) return;
        const int t1 = (int)min64((int64_t)n_rows, (int64_t)tk + chunk);
        for (int t = (int)tk; t < t1; ++t) {
            const int64_t b = row_ptr[t];
            const int k = (int)(row_ptr[t + 1] - b);
            const float yt = y[t];
            bool ok = true;
            float acc = 0.0f;
            if (k <= 32 * R) {
                int j[R];
                float x[R], wv[R];
                long long rank[R];
#pragma unroll
                for (int r = 0; r < R; ++r) {
                    const int i = r * 32 + lane;
                    j[r] = i < k ? col[b + i] : 0;
                    x[r] = i < k ? (val ? val[b + i] : 1.0f) : 0.0f;
                    rank[r] = i < k ? (long long)(gate[b + i] & GATE_RANK) : 0;
                    wv[r] = 0.0f;
                }
#pragma unroll
                for (int r = 0; r < R; ++r)
                    if (r * 32 + lane < k && ok) {
                        if constexpr (PREFIX)
                            ok = read_prefix(w, wbits, writes, rbits, feat_ptr, j[r], rank[r], rank[r] - delay, wv[r],
                                             status, timeout);
                        else
                            ok = read_admitted(w, writes, reads, j[r], rank[r] - delay, wv[r], status, timeout);
                    }
                if (!__all_sync(FULL, ok)) return;
                trace_mark(trace, trace_base + t, 0);
#pragma unroll
                for (int r = 0; r < R; ++r)
                    if (r * 32 + lane < k) acc = __fmaf_rn(wv[r], x[r], acc);
                const float m = warp_combine(acc);
                const float c = __fmul_rn(eta, dev_grad(loss, m, yt));
                trace_mark(trace, trace_base + t, 1);   // before any write is visible
                if (coef && lane == 0) coef[t] = c;
#pragma unroll
                for (int r = 0; r < R; ++r)
                    if (r * 32 + lane < k && ok) {
                        if constexpr (PREFIX)
                            ok = write_prefix(w, wbits, rbits, reads, feat_ptr, j[r], rank[r], rank[r] - delay + 1,
                                              __fmul_rn(c, x[r]), status, timeout);
                        else
                            ok = write_admitted(w, writes, reads, j[r], rank[r] - delay + 1, __fmul_rn(c, x[r]),
                                                status, timeout);
                    }
                if (!__all_sync(FULL, ok)) return;
                continue;
            }
            // long example: element by element
            for (int i = lane; i < k && ok; i += 32) {
                const int jj = col[b + i];
                const long long rk = (long long)(gate[b + i] & GATE_RANK);
                float v1 = 0.0f;
                if constexpr (PREFIX)
                    ok = read_prefix(w, wbits, writes, rbits, feat_ptr, jj, rk, rk - delay, v1, status, timeout);
                else
                    ok = read_admitted(w, writes, reads, jj, rk - delay, v1, status, timeout);
                if (ok) acc = __fmaf_rn(v1, val ? val[b + i] : 1.0f, acc);
            }
            if (!__all_sync(FULL, ok)) return;
            trace_mark(trace, trace_base + t, 0);
            const float m = warp_combine(acc);
            const float c = __fmul_rn(eta, dev_grad(loss, m, yt));
            trace_mark(trace, trace_base + t, 1);   // before any write is visible
            if (coef && lane == 0) coef[t] = c;
            for (int i = lane; i < k && ok; i += 32) {
                const int jj = col[b + i];
                const long long rk = (long long)(gate[b + i] & GATE_RANK);
                const float step = __fmul_rn(c, val ? val[b + i] : 1.0f);
                if constexpr (PREFIX)
                    ok = write_prefix(w, wbits, rbits, reads, feat_ptr, jj, rk, rk - delay + 1, step, status, timeout);
                else
                    ok = write_admitted(w, writes, reads, jj, rk - delay + 1, step, status, timeout);
            }
            if (!__all_sync(FULL, ok)) return;
        }
    }
}

}  // namespace

namespace pdb {

int ssp_run(const pdb_csr *X, const float *y, const uint32_t *gate, float *w, unsigned *writes, unsigned *reads,
            unsigned long long *ticket, long long delay, float *coef, int loss, float eta, int n_epochs, int width,
            const pdb_opts *opts, int *status, uint64_t timeout, cudaStream_t s, const int64_t *feat_ptr,
            unsigned *rbits, unsigned *wbits, int64_t n_words)
{
    const int32_t n = (int32_t)X->n_rows;
    const int64_t F = X->n_cols;
    const int chunk = (opts && opts->ticket_chunk > 0) ? opts->ticket_chunk : 2;
    const bool prefix = rbits != nullptr;
    auto kern = prefix ? (width == 2 ? k_sgd_ssp<2, true> : width == 4 ? k_sgd_ssp<4, true> : k_sgd_ssp<8, true>)
                       : (width == 2 ? k_sgd_ssp<2, false> : width == 4 ? k_sgd_ssp<4, false> : k_sgd_ssp<8, false>);
    const int grid = persistent_grid((const void *)kern, opts);
    for (int ep = 0; ep < n_epochs; ++ep) {
        int rc = fill_words(writes, 0u, sizeof(unsigned) * (size_t)F, s);
        rc = rc ? rc : fill_words(reads, 0u, sizeof(unsigned) * (size_t)F, s);
        if (prefix) {
            rc = rc ? rc : fill_words(rbits, 0u, sizeof(unsigned) * (size_t)n_words, s);
            rc = rc ? rc : fill_words(wbits, 0u, sizeof(unsigned) * (size_t)n_words, s);
        }
        rc = rc ? rc : fill_words(ticket, 0u, sizeof(unsigned long long), s);
        if (rc != PDB_OK) return rc;
        kern<<<grid, THREADS, 0, s>>>(n, X->row_ptr, X->col, X->val, y, gate, w, writes, reads, delay,
                                      coef ? coef + (int64_t)ep * n : nullptr, loss, eta, ticket, chunk, status,
                                      timeout, opts ? opts->trace : nullptr, (int64_t)ep * n, feat_ptr, rbits, wbits);
        note_launch();
    }
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

}  // namespace pdb
