// Internal helpers shared by the libpdb translation units: status words,
// acquire/release memory operations, bounded waits, the grid barrier of the
// persistent kernels, the fp32 numerics of one SGD transaction, and the
// handle layouts.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "pdb.h"

namespace pdb {

constexpr unsigned FULL = 0xffffffffu;
constexpr int THREADS = 256;             // block size of every persistent kernel
constexpr int WARPS = THREADS / 32;

// ------------------------------------------------------------------ host
struct Launch {
    int sms = 0;
    int device = 0;
};
Launch launch_info();
int occupancy_blocks(const void *kernel, int threads, size_t smem);
int persistent_grid(const void *kernel, const pdb_opts *opts);
uint64_t timeout_ns(const pdb_opts *opts);
int alloc(void **p, size_t bytes, cudaStream_t s);   // stream-ordered, 256-byte aligned
void release(void *p, cudaStream_t s);
cudaStream_t own_stream();                           // the library's non-blocking stream (current device)
int bits_for(int64_t max_key);                        // bits to hold values 0..max_key (>= 1)
int grid_1d(int64_t n);                               // blocks of 256 threads for a grid-stride loop

// chain engine (chain.cu)
int chain_max_row();
int64_t resident_smem(int64_t n_cols, int64_t max_row);   // 0 when the weights do not fit in one block
int64_t block_ready_smem(int64_t n_cols, int64_t max_row);   // 0 when the records do not fit in one block
int block_ready_run(const pdb_csr *X, const float *y, const uint32_t *gate, float *w, int loss, float eta,
                    int epochs, int max_row, int *status, uint64_t timeout, uint64_t *trace, cudaStream_t s);
int resident_run(const pdb_csr *X, const float *y, float *w, int loss, float eta, int epochs, int max_row,
                 int *status, uint64_t *trace, cudaStream_t s);
int chain_schedule(const int32_t *prev, const int32_t *next, const int32_t *row_of, const int64_t *row_ptr,
                   int64_t nnz, int64_t max_row, uint32_t *link, const int *status, cudaStream_t s);
int chain_run(const pdb_csr *X, const float *y, const uint32_t *link, float *w, int loss, float eta, int epochs,
              int max_row, int *status, uint64_t *trace, cudaStream_t s);
void note_launch();                                   // count one kernel launch (pdb_launch_count)

// counters that many blocks add to are spread over this many words (summed by the reader)
constexpr int DESC_SPREAD = 32;

// Stable LSD radix sort of (key, value) pairs, digits of 8 to 10 bits.
// vals_in == nullptr means value = index.  Sorted pairs land in
// keys_out/vals_out; keys_tmp/vals_tmp are scratch of n elements each.
// Kernels return early when *status != 0.  With range != 0 every key must be
// below it (else PDB_ERANGE in *status); with descents != nullptr the
// DESC_SPREAD device counters there gain, summed, the number of i >= 1 with
// (int32) key[i-1] >= (int32) key[i] (both during the first read of the keys).
int radix_sort(const uint32_t *keys_in, const int32_t *vals_in, uint32_t *keys_out, int32_t *vals_out,
               uint32_t *keys_tmp, int32_t *vals_tmp, int64_t n, int key_bits, const int *status,
               cudaStream_t s, uint32_t range = 0, int *descents = nullptr);
// stable sort on key bits [lo_bit, hi_bit) only (the bits below stay in input order)
int radix_sort_bits(const uint32_t *keys_in, const int32_t *vals_in, uint32_t *keys_out, int32_t *vals_out,
                    uint32_t *keys_tmp, int32_t *vals_tmp, int64_t n, int lo_bit, int hi_bit, const int *status,
                    cudaStream_t s);

// ptr[k] = first index i of the sorted keys with keys[i] >= k, k = 0..n_bins
// (n_bins read from *n_bins_dev when that is non-null).
int segment_bounds(const uint32_t *sorted_keys, int64_t n, int64_t n_bins, const int *n_bins_dev, int64_t *ptr,
                   const int *status, cudaStream_t s);

// ------------------------------------------------------------------ device
__host__ __device__ __forceinline__ int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }
__device__ __forceinline__ void set_status(int *st, int code) { atomicCAS(st, 0, code); }
__device__ __forceinline__ int read_status(const int *st) { return *(volatile const int *)st; }

__device__ __forceinline__ unsigned ld_acquire(const unsigned *p)
{
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_release(unsigned *p, unsigned v)
{
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ int ld_acquire_i(const int *p)
{
    int v;
    asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ uint64_t globaltimer()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ unsigned lanemask_lt()
{
    unsigned m;
    asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
    return m;
}

// Grid barrier for cooperative (co-resident) launches.  Generation counter:
// read the generation, arrive, the last arriver resets the count and bumps
// the generation; the others wait for the bump.  Every wait is bounded by
// `deadline` (globaltimer ns) and gives up early when the status word is
// set, so a failed block cannot hang the rest.  Returns false on give-up.
struct GridBarrier {
    unsigned count;
    unsigned gen;
};

// snap_src/snap_dst (optional): the last arriver copies *snap_src into
// *snap_dst before it releases the others, so every block reads one value
// that no block can change until the next barrier.
__device__ __forceinline__ bool grid_sync(GridBarrier *bar, int *status, uint64_t timeout, int *snap_src = nullptr,
                                          int *snap_dst = nullptr)
{
    __shared__ int s_ok;
    __syncthreads();
    if (threadIdx.x == 0) {
        int ok = 1;
        unsigned gen = ld_acquire(&bar->gen);
        __threadfence();
        unsigned arrived = atomicAdd(&bar->count, 1u);
        if (arrived == gridDim.x - 1) {
            if (snap_src) *(volatile int *)snap_dst = atomicAdd(snap_src, 0);
            atomicExch(&bar->count, 0u);
            __threadfence();
            st_release(&bar->gen, gen + 1);
        } else {
            uint64_t t0 = globaltimer();
            unsigned spins = 0;
            while (ld_acquire(&bar->gen) == gen) {
                if ((++spins & 63u) == 0) {
                    if (read_status(status) != 0) { ok = 0; break; }
                    if (globaltimer() - t0 > timeout) { set_status(status, PDB_ETIMEOUT); ok = 0; break; }
                }
                __nanosleep(32);
            }
        }
        __threadfence();
        s_ok = ok && read_status(status) == 0;
    }
    __syncthreads();
    return s_ok != 0;
}

// ------------------------------------------------------------------ numerics
// e^x: Cody-Waite argument reduction x = k ln2 + r with k = rint(x log2e)
// (W. J. Cody and W. Waite, Software Manual for the Elementary Functions,
// 1980); ln2 is split into a head with 16 significant bits, so k*head is
// exact for |k| <= 256 and x - k*head is exact (Sterbenz), and a tail.  e^r
// is the degree-7 Taylor polynomial sum r^n/n! in Horner form with fused
// multiply-adds (|r| <= 0.35: truncation below 1e-8 relative).  2^k is
// applied as two exact power-of-two factors so the one rounding happens in
// the final product, also for subnormal results.  Inputs are clamped to
// [-104, 89], where the result has already underflowed to 0 / overflowed.
// rint and the conversion of k to an integer both come from one exact
// addition of 1.5 * 2^23 (|x log2e| < 2^22: the sum's last mantissa bits are
// k, rounded to nearest even); a NaN input is returned at the end, so the
// path has no branch (the clamp, a min and a max, maps NaN to -104 on the
// way).  k*head is exact, so x - k*head is one fused multiply-add.
__device__ __forceinline__ float dev_expf(float x0)
{
    const float x = fminf(fmaxf(x0, -104.0f), 89.0f);
    const float log2e = 1.44269502162933349609375f;      // nearest float to log2(e)
    const float ln2_head = 0.693145751953125f;           // 45426 * 2^-16
    const float ln2_tail = 1.428606765330187045e-06f;     // ln2 - head, rounded to float
    const float shifter = 12582912.0f;                    // 1.5 * 2^23
    const float u = __fadd_rn(__fmul_rn(x, log2e), shifter);
    const float kf = __fsub_rn(u, shifter);
    const int k = __float_as_int(u) - 0x4B400000;
    float r = __fmaf_rn(-kf, ln2_head, x);
    r = __fsub_rn(r, __fmul_rn(kf, ln2_tail));
    float p = 1.0f / 5040.0f;
    p = __fmaf_rn(p, r, 1.0f / 720.0f);
    p = __fmaf_rn(p, r, 1.0f / 120.0f);
    p = __fmaf_rn(p, r, 1.0f / 24.0f);
    p = __fmaf_rn(p, r, 1.0f / 6.0f);
    p = __fmaf_rn(p, r, 0.5f);
    p = __fmaf_rn(p, r, 1.0f);
    p = __fmaf_rn(p, r, 1.0f);
    const int h = k / 2;
    const int k2 = k - h;
    const float s1 = __int_as_float((h + 127) << 23);
    const float s2 = __int_as_float((k2 + 127) << 23);
    // with 0.7 < p < 1.5 and -125 <= k <= 127, p * 2^k is normal, so one exact
    // scaling by 2^k equals the two-factor form (which the rest of the range needs)
    const float sk = __int_as_float((k + 127) << 23);
    const float e = k >= -125 && k <= 127 ? __fmul_rn(p, sk) : __fmul_rn(__fmul_rn(p, s1), s2);
    return x0 != x0 ? x0 : e;
}

// execution trace (pdb_opts.trace): lane 0 stamps %globaltimer into
// trace[2 * idx + which] (idx = epoch * n_rows + example), which = 0 once
// every weight the example reads has been read, which = 1 once its update is
// computed and before any of its writes is issued.  Called by the whole warp;
// the __syncwarp keeps the other lanes' later writes after the stamp.
__device__ __forceinline__ void trace_mark(uint64_t *trace, int64_t idx, int which)
{
    if (trace) {
        if ((threadIdx.x & 31) == 0) trace[2 * idx + which] = globaltimer();
        __syncwarp();
    }
}

// 1/d rounded to nearest for 1 <= d < 2^126: Newton-Raphson from the
// hardware's approximate reciprocal, then one step with the exact residual
// 1 - d*y1 (P. Markstein, "Computation of elementary functions on the IBM
// RISC System/6000 processor", IBM J. Res. Dev. 34(1), 1990).  Equal to the
// IEEE quotient 1/d for every float d in that range (checked exhaustively on
// the GPU); shorter on the dependent path than the general division.
__device__ __forceinline__ float recip_ge1(float d)
{
    float y0;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y0) : "f"(d));
    const float e = __fmaf_rn(-d, y0, 1.0f);
    const float y1 = __fmaf_rn(y0, e, y0);
    const float r = __fmaf_rn(-d, y1, 1.0f);
    return __fmaf_rn(y1, r, y1);
}

// derivative of the example's loss with respect to its margin m; for the
// logistic loss with y = +1 or -1, -y/d = -y * (1/d) exactly (rounding to
// nearest is symmetric), so the reciprocal above gives the IEEE quotient's
// bits.  The reciprocal is formed unconditionally and the division taken only
// outside its range, so the common path has no branch.
__device__ __forceinline__ float dev_grad(int loss, float m, float y)
{
    if (loss == PDB_LOSS_LOGISTIC) {
        const float d = __fadd_rn(1.0f, dev_expf(__fmul_rn(y, m)));
        const float q = recip_ge1(d);
        float g = y > 0.0f ? -q : q;
        if (!((y == 1.0f || y == -1.0f) && d < 0x1p126f)) g = __fdiv_rn(-y, d);
        return g;
    }
    if (loss == PDB_LOSS_SQUARED) return __fsub_rn(m, y);
    return __fmul_rn(y, m) < 1.0f ? -y : 0.0f;
}

// the step size times the derivative, eta * dev_grad(loss, m, y), with the
// same bits: on the reciprocal path eta * (-y q) = (-y eta) * q exactly, so
// the sign goes on eta, which is known before m
__device__ __forceinline__ float dev_step(int loss, float m, float y, float eta)
{
    if (loss == PDB_LOSS_LOGISTIC) {
        const float d = __fadd_rn(1.0f, dev_expf(__fmul_rn(y, m)));
        float c = __fmul_rn(y > 0.0f ? -eta : eta, recip_ge1(d));
        if (!((y == 1.0f || y == -1.0f) && d < 0x1p126f)) c = __fmul_rn(eta, __fdiv_rn(-y, d));
        return c;
    }
    return __fmul_rn(eta, dev_grad(loss, m, y));
}

// combine the 32 lane partial sums pairwise: xor 16, 8, 4, 2, 1 (every lane
// ends with the same value because fp32 addition commutes)
__device__ __forceinline__ float warp_combine(float a)
{
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) a = __fadd_rn(a, __shfl_xor_sync(FULL, a, off));
    return a;
}

// Gate word of a position (the conflicts' per-position schedule input):
// bits 0..28 occurrence rank of its feature, bit 29 the next occurrence lies
// within `near` positions, bit 30 the previous one does, bit 31 last
// occurrence of the feature.
constexpr uint32_t GATE_RANK = 0x1fffffffu;
constexpr uint32_t GATE_NEAR_NEXT = 1u << 29;
constexpr uint32_t GATE_NEAR_PREV = 1u << 30;
constexpr uint32_t GATE_LAST = 1u << 31;

// WINDOW engine control block (device), zeroed before every epoch
struct WindowCtl {
    unsigned long long ticket;  // next example to hand out
    long long wpos;             // every example starting below this position has finished
    unsigned arrive;            // blocks started so far (the first one sweeps)
    unsigned pad;
};

// admissible delay; rbits == nullptr selects the counting gates, else the
// prefix gates on the done-bitmaps rbits / wbits (n_words words each)
int ssp_run(const pdb_csr *X, const float *y, const uint32_t *gate, float *w, unsigned *writes, unsigned *reads,
            unsigned long long *ticket, long long delay, float *coef, int loss, float eta, int n_epochs, int width,
            const pdb_opts *opts, int *status, uint64_t timeout, cudaStream_t s, const int64_t *feat_ptr,
            unsigned *rbits, unsigned *wbits, int64_t n_words);

int ensure_row_of(pdb_conflicts *c, cudaStream_t s);   // builds c->row_of on first use (stream-ordered)

int window_run(const pdb_csr *X, const float *y, const uint32_t *gate, float *w, unsigned long long *rec,
               unsigned *epoch_count, unsigned *done, int64_t done_cap, WindowCtl *ctl, int64_t near, int loss,
               float eta, int n_epochs, int width, const pdb_opts *opts, int *status, uint64_t timeout,
               cudaStream_t s);

}  // namespace pdb

// ------------------------------------------------------------------ handles
struct pdb_conflicts {
    int device;
    int64_t n_rows, n_cols, nnz;
    const int64_t *row_ptr;  // the caller's D (immutable, must outlive the handle)
    const int32_t *col;
    const float *val;
    int32_t *csc_pos;        // positions grouped by feature, data order inside a feature
    int64_t *feat_ptr;       // [F+1]
    uint32_t *gate;          // per position: occurrence rank and flags (GATE_* below); above 2^22
                             // positions built on first use (build.cu) from gate_sorted
    uint32_t *gate_sorted;   // above 2^22 positions: the gate words in csc_pos order
    uint32_t *gate_window;   // the WINDOW engine's gate: above 2^22 positions only the words of
                             // positions with a near pair (0 elsewhere), else = gate
    int64_t near;            // distance (positions) under which an occurrence pair counts as near
    int32_t *row_of;         // example of each position (built on first use)
    int32_t *prev, *next, *rank;  // materialized from the above on first request
    int32_t *npred;          // per example: occurrences with an earlier occurrence (LEVELS)
    int *info;               // device: [0] status, [1] max chain, [2] longest row, [3] any unsorted row,
                             // [4] near occurrence pairs
    int *h_info;             // pinned host copy of info, filled at the end of the build
    cudaEvent_t ev0, ev1, ev_sgd0, ev_sgd1, ev_bsp0, ev_bsp1, ev_k0, ev_k1;
    cudaEvent_t ev_use;      // recorded after the last work any call enqueued on the handle
    bool timed_build, timed_sgd, timed_bsp;
    int *status;             // = info (first error recorded by a kernel)
};

struct LevelCtl {
    int tail;                 // frontier queue length
    int n_levels;             // L
    int max_width;
    int end;                  // frontier end snapshot taken at each grid barrier
    pdb::GridBarrier bar;
};

struct pdb_schedule {
    const pdb_conflicts *c;
    pdb_sched_mode mode;
    int32_t *level, *order, *indeg, *queue;
    int64_t *level_ptr;
    LevelCtl *ctl;            // device
    unsigned long long *rec;  // READY: per feature (weight bits | version << 32); WINDOW: near hand-offs
    unsigned *reads, *writes; // READY under pdb_ssp_epoch: reads / writes of each feature this epoch (first use);
                              // under prefix gates the known-done prefix of each feature's reads / writes
    unsigned *rbits, *wbits;  // READY under pdb_ssp_epoch with prefix gates: done-bitmaps over the CSC slots
    uint32_t *link;           // CHAIN: per position, receive flag and push target
    bool resident;            // CHAIN: weights resident in shared memory (no link words)
    unsigned epochs_run;      // WINDOW: epochs run so far (epoch stamp of the record tags, done-flag tag)
    unsigned *prog;           // WINDOW: done flag per chunk of examples (zeroed once)
    int64_t prog_cap;         // WINDOW: flags allocated (one per example: chunks of one example or more)
    pdb::WindowCtl *wctl;     // WINDOW: ticket and watermark
    pdb::GridBarrier *bar;    // barrier for the level-synchronous engine
    unsigned long long *ticket;
    cudaEvent_t ev0, ev1;
    cudaEvent_t ev_use;      // recorded after the last work any call enqueued on the handle
    bool timed;
};

// BSP batches for the data-parallel split (pdb_bsp_plan_build): every pair of
// the data sorted by (batch, feature, example), with its feature, example and
// value, and where each batch's pairs start (device and host copies)
struct pdb_bsp_plan {
    const pdb_conflicts *c;
    int64_t batch, n_batches;
    int64_t *bptr;            // [n_batches + 1] device
    int64_t *h_bptr;          // [n_batches + 1] host
    int32_t *bcol, *brow;
    cudaEvent_t ev_use;       // recorded after the last work any call enqueued on the plan
    float *bval;
};

namespace pdb {
// Handles record ev_use on the call's stream after every call that enqueues
// work on them; freeing a handle waits for that event only (not for the whole
// device, where other streams may be busy), then returns its arrays to the
// pool.
void mark_use(const pdb_conflicts *c, const pdb_schedule *h, cudaStream_t s);
// records ev_use of the handles on the call's stream when the call returns
// (every return path, after everything the call enqueued)
struct UseMark {
    const pdb_conflicts *c;
    const pdb_schedule *h;
    cudaStream_t s;
    ~UseMark() { mark_use(c, h, s); }
};
// host-side pinned words for a conflicts handle's info copy, from a slab that
// is kept for the process (freeing pinned memory would synchronize the device)
// fill bytes / 4 words at p with v on s by a kernel (a memset may run on a
// copy engine and queue behind the caller's copies); bytes a multiple of 4
int fill_words(void *p, uint32_t v, size_t bytes, cudaStream_t s);
int *info_slot_take();
void info_slot_give(int *slot);

// Scope of one C-ABI call: an NVTX range named after the call (shown by
// profilers, a no-op without one), and, when the environment variable
// PDB_LOG is set to anything but "" or "0", one line of pdb_get_stats on
// stderr after the call (pdb_get_stats synchronizes the device, so this is a
// debugging aid).  pc / ph point at a handle the call creates, read when the
// scope ends.
struct ApiScope {
    const char *name;
    const pdb_conflicts *c;
    const pdb_schedule *h;
    pdb_conflicts *const *pc;
    pdb_schedule *const *ph;
    bool log;
    ApiScope(const char *name_, const pdb_conflicts *c_, const pdb_schedule *h_ = nullptr,
             pdb_conflicts *const *pc_ = nullptr, pdb_schedule *const *ph_ = nullptr, bool log_ = true);
    ~ApiScope();
    ApiScope(const ApiScope &) = delete;
    ApiScope &operator=(const ApiScope &) = delete;
};
}  // namespace pdb
