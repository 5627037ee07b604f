// Window engine: pdb_sgd_epoch under a WINDOW schedule.
//
// When consecutive occurrences of a feature mostly lie far apart in the data
// (ids drawn from many more features than one batch of concurrent examples
// touches), almost every Read Constraint of Section 4.4 is already met by the
// time an example runs: the previous writer finished long ago.  This engine
// pays for the constraint only where it can bind:
//
//   * a position whose previous occurrence lies at least `near` positions
//     back ("far") reads w_j from the plain fp32 array, once the example has
//     seen the completion watermark pass that distance: every example below
//     the watermark has finished and its writes are visible;
//   * a position whose previous occurrence lies closer ("near", gate bit 30)
//     takes the weight from that occurrence through a 64-bit record of
//     feature j, bits(w_j) | tag << 32, as under READY (the read protocol of
//     Section 5): one load both checks the tag and returns the weight.  The
//     tag is the reader's occurrence rank plus an epoch stamp in bits 29-31,
//     so records left by an earlier epoch never match and need no reset.
//
// Each position writes its new weight exactly once: into the record when its
// next occurrence is near (gate bit 29; the near reader takes it from
// there), else into w_j (read by a far successor, or final).  So w_j always
// holds the weight of the latest writer whose successor is far, which is the
// one a far reader needs; no position pays for both.
//
// Watermark: examples are taken in data order from a ticket counter, a
// chunk of consecutive ones per warp.  When a warp has finished chunk c it
// sets done[c] to the epoch's tag (release, after a fence that covers the
// chunk's weight stores); it does so right after issuing the first loads of
// its next chunk, or before it exits.  The tag is unique to the epoch (a
// 32-bit count of the schedule's epochs), so flags of earlier epochs never
// count and the array is zeroed only once.  One block sweeps: the first
// block of the grid to start (an arrival counter, not blockIdx, picks it,
// so it is running whichever blocks the device has made resident).  It
// scans done[] from the current watermark and publishes the first position
// of the first unfinished chunk as `wpos` (release).  An example refreshes
// its view of `wpos` with one acquire load issued while its ids and values
// are still in flight.
//
// Deadlock freedom, with any subset of the grid resident: a chunk is only
// ever held by a warp that is running (it took the ticket).  The oldest
// unfinished chunk waits for nothing -- its near predecessors are finished,
// and its watermark condition is capped at the first position of its own
// chunk, which the watermark reaches once every earlier chunk has set its
// flag.  Those flags are set without waiting, and the sweeper is running.
// Blocks the device has not started yet hold no chunk and hold nothing
// back.  Every wait, including the sweeper's, is bounded by the timeout.
#include <cuda_runtime.h>

#include "common.cuh"

using namespace pdb;

namespace {

__device__ __forceinline__ long long ld_acquire_s64(const long long *p)
{
    long long v;
    asm volatile("ld.acquire.gpu.global.s64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ unsigned long long ld_rec(const unsigned long long *p)
{
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_rec(unsigned long long *p, float w, unsigned tag)
{
    const unsigned long long v = (unsigned long long)__float_as_uint(w) | ((unsigned long long)tag << 32);
    asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ void fence_acq_rel() { asm volatile("fence.acq_rel.gpu;" ::: "memory"); }

// Weight accesses carry an L2 evict_last policy: the streamed ids, values and
// gate words are read once, so the L2 keeps weights in their place (a weight
// line is used again by its read-modify-write and by any other feature of the
// line before it leaves).  Measured on the low-conflict access pattern: ~5%
// less time than plain cache-global accesses.
__device__ __forceinline__ uint64_t policy_evict_last()
{
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ float ld_w(const float *a, uint64_t pol)
{
    float v;
    asm volatile("ld.global.L1::no_allocate.L2::cache_hint.f32 %0, [%1], %2;" : "=f"(v) : "l"(a), "l"(pol) : "memory");
    return v;
}
__device__ __forceinline__ void st_w(float *a, float v, uint64_t pol)
{
    asm volatile("st.global.L1::no_allocate.L2::cache_hint.f32 [%0], %1, %2;" ::"l"(a), "f"(v), "l"(pol) : "memory");
}
__device__ __forceinline__ void max_release(long long *p, long long v)
{
    asm volatile("red.release.gpu.global.max.s64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

// gives up when the failure is elsewhere (status set) or the wait ran out
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

// Waits until the watermark has reached `need` (positions) or gives up.
// `known` holds this lane's last acquired watermark (it only grows).
__device__ __noinline__ bool wait_watermark(const WindowCtl *ctl, long long need, long long &known, int *status,
                                            uint64_t timeout)
{
    const uint64_t t0 = globaltimer();
    unsigned spins = 0, nap = 64;
    while (known < need) {
        __nanosleep(nap);
        nap = nap < 1024 ? 2 * nap : 1024;
        known = ld_acquire_s64(&ctl->wpos);
        if (known < need && !keep_waiting(spins, t0, status, timeout)) return false;
    }
    return true;
}

// Gathers this lane's weights: far ones from w (their watermark condition
// already checked), near ones from the records, waiting for each wanted tag.
template <int R>
__device__ __forceinline__ bool gather_window(const float *w, const unsigned long long *rec, const int *j,
                                              const uint32_t *g, unsigned stamp, float *wv, int lane, int k,
                                              int *status, uint64_t timeout, uint64_t pol)
{
    unsigned pending = 0;
#pragma unroll
    for (int r = 0; r < R; ++r) {
        wv[r] = 0.0f;
        if (r * 32 + lane < k) {
            if (g[r] & GATE_NEAR_PREV) {
                const unsigned long long v = ld_rec(rec + j[r]);
                wv[r] = __uint_as_float((unsigned)v);
                if ((unsigned)(v >> 32) != ((g[r] & GATE_RANK) | stamp)) pending |= 1u << r;
            } else {
                wv[r] = ld_w(w + j[r], pol);
            }
        }
    }
    if (pending == 0) return true;
    const uint64_t t0 = globaltimer();
    unsigned spins = 0, nap = 32;
    while (pending) {
        __nanosleep(nap);
        nap = nap < 512 ? 2 * nap : 512;
#pragma unroll
        for (int r = 0; r < R; ++r)
            if (pending & (1u << r)) {
                const unsigned long long v = ld_rec(rec + j[r]);
                if ((unsigned)(v >> 32) == ((g[r] & GATE_RANK) | stamp)) {
                    wv[r] = __uint_as_float((unsigned)v);
                    pending &= ~(1u << r);
                }
            }
        if (pending && !keep_waiting(spins, t0, status, timeout)) return false;
    }
    return true;
}

// the new weight goes where the next occurrence will look for it
__device__ __forceinline__ void publish(int j, uint32_t g, float nw, float *w, unsigned long long *rec,
                                        unsigned stamp, uint64_t pol)
{
    if (g & GATE_NEAR_NEXT)
        st_rec(rec + j, nw, ((g & GATE_RANK) + 1u) | stamp);
    else
        st_w(w + j, nw, pol);
}

// no near previous occurrence (far, or none at all): read from w after the
// watermark; the gate of such a position may carry no rank (inputs above
// 2^22 positions keep only the near pairs' words), and the watermark
// condition holds for a first occurrence too
__device__ __forceinline__ bool is_far(uint32_t g) { return !(g & GATE_NEAR_PREV); }

// chunk finished: every lane's weight stores are visible before the flag
// (fence by every lane, then one store by lane 0)
__device__ __forceinline__ void publish_done(unsigned *flag, unsigned tag)
{
    fence_acq_rel();
    __syncwarp();
    if ((threadIdx.x & 31) == 0) st_release(flag, tag);
}

// One example.  The first example of a chunk sets the done flag of the
// warp's previous chunk (flag != nullptr) right after issuing its ids and
// values: the fence then waits for that chunk's weight stores while these
// loads are in flight anyway.
template <int R>
__device__ __forceinline__ bool window_example(int t, int64_t floor_pos, const int64_t *__restrict__ row_ptr,
                                               const int32_t *__restrict__ col, const float *__restrict__ val,
                                               const float *__restrict__ y, const uint32_t *__restrict__ gate,
                                               float *w, unsigned long long *rec, unsigned stamp,
                                               const WindowCtl *ctl, int64_t near, int loss, float eta,
                                               long long &known, unsigned *flag, unsigned tag, int *status,
                                               uint64_t timeout, uint64_t *trace, int64_t idx, uint64_t pol)
{
    const int lane = threadIdx.x & 31;
    const int64_t b = row_ptr[t];
    const int k = (int)(row_ptr[t + 1] - b);
    const float yt = y[t];
    // a far previous occurrence sits at or before p - near (p < b + k) and
    // before this example's chunk: below `need`
    const long long need = (long long)min64(floor_pos, b + k - near);
    if (k <= 32 * R) {
        int j[R];
        float x[R], wv[R];
        uint32_t g[R];
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int i = r * 32 + lane;
            j[r] = i < k ? __ldcs(col + b + i) : 0;
            x[r] = i < k ? (val ? __ldcs(val + b + i) : 1.0f) : 0.0f;
            g[r] = i < k ? __ldcs(gate + b + i) : 0u;
        }
        if (flag) publish_done(flag, tag);
        // refresh the watermark while the loads above are in flight
        if (known < need) known = ld_acquire_s64(&ctl->wpos);
        bool far = false;
#pragma unroll
        for (int r = 0; r < R; ++r) far |= r * 32 + lane < k && is_far(g[r]);
        bool ok = !far || known >= need || wait_watermark(ctl, need, known, status, timeout);
        ok = ok && gather_window<R>(w, rec, j, g, stamp, wv, lane, k, status, timeout, pol);
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
            if (r * 32 + lane < k) publish(j[r], g[r], __fsub_rn(wv[r], __fmul_rn(c, x[r])), w, rec, stamp, pol);
        __syncwarp();   // the next example of the chunk may read these weights from another lane
        return true;
    }
    // long example: gather element by element, then a second pass (no other
    // example writes these features before this one does, so the second
    // read of w or of a record returns the same weight)
    if (flag) publish_done(flag, tag);
    if (known < need) known = ld_acquire_s64(&ctl->wpos);
    float acc = 0.0f;
    bool ok = true;
    for (int i = lane; i < k && ok; i += 32) {
        const int jj[1] = {col[b + i]};
        const uint32_t gg[1] = {gate[b + i]};
        float v1[1];
        ok = !is_far(gg[0]) || known >= need || wait_watermark(ctl, need, known, status, timeout);
        ok = ok && gather_window<1>(w, rec, jj, gg, stamp, v1, 0, 1, status, timeout, pol);
        if (ok) acc = __fmaf_rn(v1[0], val ? val[b + i] : 1.0f, acc);
    }
    if (!__all_sync(FULL, ok)) return false;
    trace_mark(trace, idx, 0);
    const float m = warp_combine(acc);
    const float c = __fmul_rn(eta, dev_grad(loss, m, yt));
    trace_mark(trace, idx, 1);   // before any write is visible
    for (int i = lane; i < k; i += 32) {
        const int jj = col[b + i];
        const uint32_t gg = gate[b + i];
        const float xx = val ? val[b + i] : 1.0f;
        const float wo = (gg & GATE_NEAR_PREV) ? __uint_as_float((unsigned)ld_rec(rec + jj)) : ld_w(w + jj, pol);
        publish(jj, gg, __fsub_rn(wo, __fmul_rn(c, xx)), w, rec, stamp, pol);
    }
    __syncwarp();
    return true;
}

// The sweeping block: scan the done flags from the watermark's chunk,
// SWEEP_SPAN of them per round (16-byte loads of four flags, the first one
// rounded down to a multiple of four; flags below the watermark count as
// set), and publish the first position of the first unfinished chunk after
// each advance.  A round costs a few memory latencies under the engine's
// load, so it must cover many chunks: the workers finish ~100 chunks per
// microsecond.  Relaxed loads then one fence: an acquire of all of them
// without serializing the loads.
constexpr int SWEEP_VEC = 8;                                    // 16-byte loads per thread and round
constexpr unsigned SWEEP_SPAN = THREADS * SWEEP_VEC * 4;        // flags per round

__device__ __forceinline__ uint4 ld_relaxed_v4(const unsigned *p)
{
    uint4 v;
    asm volatile("ld.relaxed.gpu.global.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p)
                 : "memory");
    return v;
}

__device__ void sweep(int32_t n_rows, const int64_t *__restrict__ row_ptr, const unsigned *done, unsigned tag,
                      unsigned n_chunks, int chunk, WindowCtl *ctl, int *status, uint64_t timeout)
{
    __shared__ unsigned s_first[WARPS];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    unsigned wm = 0;
    uint64_t t_last = globaltimer();
    while (wm < n_chunks) {
        const unsigned base = wm & ~3u;           // done is 256-byte aligned: base is a 16-byte boundary
        // first chunk at or above wm whose flag this thread sees unset (n_chunks if none)
        unsigned first = n_chunks;
#pragma unroll
        for (int q = 0; q < SWEEP_VEC; ++q) {
            const unsigned c0 = base + 4u * ((unsigned)q * THREADS + threadIdx.x);
            if (c0 < n_chunks) {
                const uint4 v = ld_relaxed_v4(done + c0);
                const unsigned f[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const unsigned c = c0 + e;
                    if (c >= wm && c < n_chunks && f[e] != tag) first = min(first, c);
                }
            }
        }
        fence_acq_rel();
        for (int o = 16; o >= 1; o >>= 1) first = min(first, __shfl_xor_sync(FULL, first, o));
        if (lane == 0) s_first[warp] = first;
        __syncthreads();
        unsigned nw = s_first[0];
#pragma unroll
        for (int q = 1; q < WARPS; ++q) nw = min(nw, s_first[q]);
        __syncthreads();     // s_first is rewritten by the next scan
        // every flag in [wm, nw) was seen set; past the round's span nothing was looked at
        nw = min(nw, min(n_chunks, base + SWEEP_SPAN));
        const uint64_t now = globaltimer();
        if (nw > wm) {
            wm = nw;
            if (threadIdx.x == 0) max_release(&ctl->wpos, (long long)row_ptr[min64(n_rows, (int64_t)wm * chunk)]);
            t_last = now;
            continue;
        }
        const bool timed_out = now - t_last > timeout;
        if (read_status(status) != 0 || timed_out) {
            if (threadIdx.x == 0 && timed_out) set_status(status, PDB_ETIMEOUT);
            return;
        }
        __nanosleep(256);
    }
}

template <int R>
__global__ __launch_bounds__(THREADS) void k_sgd_window(int32_t n_rows, const int64_t *__restrict__ row_ptr,
                                                        const int32_t *__restrict__ col,
                                                        const float *__restrict__ val, const float *__restrict__ y,
                                                        const uint32_t *__restrict__ gate, float *w,
                                                        unsigned long long *rec, unsigned stamp, unsigned *done,
                                                        unsigned tag, WindowCtl *ctl, int64_t near, int loss,
                                                        float eta, int chunk, int *status, uint64_t timeout,
                                                        uint64_t *trace, int64_t trace_base)
{
    if (read_status(status)) return;
    const unsigned n_chunks = (unsigned)((n_rows + (int64_t)chunk - 1) / chunk);
    __shared__ unsigned s_arrival;
    if (threadIdx.x == 0) s_arrival = atomicAdd(&ctl->arrive, 1u);
    __syncthreads();
    if (s_arrival == 0) {
        sweep(n_rows, row_ptr, done, tag, n_chunks, chunk, ctl, status, timeout);
        return;
    }
    const int lane = threadIdx.x & 31;
    const uint64_t pol = policy_evict_last();
    long long known = 0;
    unsigned prev = 0xffffffffu;   // the chunk this warp finished last, its flag not yet set
    for (;;) {
        unsigned long long tk = 0;
        if (lane == 0) tk = atomicAdd(&ctl->ticket, (unsigned long long)chunk);
        tk = __shfl_sync(FULL, tk, 0);
        if (tk >= (unsigned long long)n_rows) {
            if (prev != 0xffffffffu) publish_done(done + prev, tag);
            return;
        }
        const int t1 = (int)min64((int64_t)n_rows, (int64_t)tk + chunk);
        const int64_t floor_pos = row_ptr[tk];
        for (int t = (int)tk; t < t1; ++t)
            if (!window_example<R>(t, floor_pos, row_ptr, col, val, y, gate, w, rec, stamp, ctl, near, loss, eta,
                                   known, (t == (int)tk && prev != 0xffffffffu) ? done + prev : nullptr, tag, status,
                                   timeout, trace, trace_base + t, pol))
                return;
        prev = (unsigned)(tk / chunk);
    }
}

}  // namespace

namespace pdb {

int window_run(const pdb_csr *X, const float *y, const uint32_t *gate, float *w, unsigned long long *rec,
               unsigned *epoch_count, unsigned *done, int64_t done_cap, WindowCtl *ctl, int64_t near, int loss,
               float eta, int n_epochs, int width, const pdb_opts *opts, int *status, uint64_t timeout,
               cudaStream_t s)
{
    const int32_t n = (int32_t)X->n_rows;
    const int chunk = (opts && opts->ticket_chunk > 0) ? opts->ticket_chunk : 2;
    if ((X->n_rows + chunk - 1) / chunk > done_cap) return PDB_EFAULT;
    auto kern = width == 2 ? k_sgd_window<2> : width == 4 ? k_sgd_window<4> : k_sgd_window<8>;
    // three blocks per SM unless the caller asks otherwise: on the low-conflict
    // workload 0.75% faster than the occupancy maximum (four), measured
    pdb_opts o = opts ? *opts : pdb_opts{};
    if (o.blocks_per_sm <= 0) o.blocks_per_sm = 3;
    int grid = persistent_grid((const void *)kern, &o);
    if (grid < 2) grid = 2;                         // the sweeping block plus at least one worker block
    for (int ep = 0; ep < n_epochs; ++ep) {
        // record tags carry an epoch stamp 1..7 (bits 29-31), different in
        // consecutive epochs of this schedule, so stale records never match;
        // done flags carry the epoch's count itself (never 0, unique until
        // the count wraps at 2^32 epochs)
        const unsigned count = (*epoch_count)++;
        const unsigned stamp = (1u + count % 7u) << 29;
        const unsigned tag = count % 0xffffffffu + 1u;
        if (tag == 1u && count != 0 && fill_words(done, 0u, sizeof(unsigned) * (size_t)done_cap, s) != PDB_OK)
            return PDB_ECUDA;
        if (fill_words(ctl, 0u, sizeof(WindowCtl), s) != PDB_OK) return PDB_ECUDA;
        kern<<<grid, THREADS, 0, s>>>(n, X->row_ptr, X->col, X->val, y, gate, w, rec, stamp, done, tag, ctl, near,
                                      loss, eta, chunk, status, timeout, opts ? opts->trace : nullptr,
                                      (int64_t)ep * X->n_rows);
        note_launch();
    }
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

}  // namespace pdb
