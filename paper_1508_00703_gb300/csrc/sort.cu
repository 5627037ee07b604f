// Stable LSD radix sort of (uint32 key, int32 value) pairs and segment
// bounds of sorted keys, plus the small host helpers of libpdb.
//
// One pass per digit of 8 to 10 bits (details at the radix sort section).
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <mutex>

#include "common.cuh"

namespace pdb {

// ------------------------------------------------------------------ host helpers
Launch launch_info()
{
    Launch l;
    cudaGetDevice(&l.device);
    cudaDeviceGetAttribute(&l.sms, cudaDevAttrMultiProcessorCount, l.device);
    return l;
}

int occupancy_blocks(const void *kernel, int threads, size_t smem)
{
    int nb = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, kernel, threads, smem) != cudaSuccess) return 0;
    return nb;
}

int persistent_grid(const void *kernel, const pdb_opts *opts)
{
    Launch l = launch_info();
    int nb = occupancy_blocks(kernel, THREADS, 0);
    if (opts && opts->blocks_per_sm > 0 && opts->blocks_per_sm < nb) nb = opts->blocks_per_sm;
    if (nb < 1) nb = 1;
    return nb * l.sms;
}

uint64_t timeout_ns(const pdb_opts *opts)
{
    double s = (opts && opts->wait_timeout_s > 0) ? opts->wait_timeout_s : 2.0;
    if (s > 1e6) s = 1e6;   // keeps the nanosecond count inside uint64_t
    return (uint64_t)(s * 1e9);
}

// The library's device memory comes from a stream-ordered memory pool of
// its own, one per device, created on first use.  Its release threshold is
// raised so that freed blocks stay in the pool for the next build or
// schedule instead of going back to the driver at every synchronization.
// The device's default pool, which other code in the process may use, is
// left as it is.
static std::mutex g_pool_lock;
static cudaMemPool_t g_pool[64];

static cudaMemPool_t library_pool(int device)
{
    if (device < 0 || device >= 64) return nullptr;
    std::lock_guard<std::mutex> guard(g_pool_lock);
    if (!g_pool[device]) {
        cudaMemPoolProps props = {};
        props.allocType = cudaMemAllocationTypePinned;
        props.location.type = cudaMemLocationTypeDevice;
        props.location.id = device;
        cudaMemPool_t pool = nullptr;
        if (cudaMemPoolCreate(&pool, &props) != cudaSuccess) {
            cudaGetLastError();
            return nullptr;
        }
        uint64_t keep = UINT64_MAX;
        cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &keep);
        g_pool[device] = pool;
    }
    return g_pool[device];
}

// The library's own non-blocking stream per device, for work that belongs to
// no caller stream: small reads of handle words and the frees of idle arrays.
static std::mutex g_own_lock;
static cudaStream_t g_own_stream[64];

cudaStream_t own_stream()
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    std::lock_guard<std::mutex> guard(g_own_lock);
    if (!g_own_stream[dev] && cudaStreamCreateWithFlags(&g_own_stream[dev], cudaStreamNonBlocking) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    return g_own_stream[dev];
}

int alloc(void **p, size_t bytes, cudaStream_t s)
{
    *p = nullptr;
    int dev = 0;
    cudaGetDevice(&dev);
    cudaMemPool_t pool = library_pool(dev);
    if (!pool) return PDB_ENOMEM;
    if (bytes == 0) bytes = 256;
    bytes = (bytes + 255) & ~(size_t)255;
    if (cudaMallocFromPoolAsync(p, bytes, pool, s) != cudaSuccess) {
        cudaGetLastError();
        *p = nullptr;
        return PDB_ENOMEM;
    }
    return PDB_OK;
}

void release(void *p, cudaStream_t s)
{
    if (p) cudaFreeAsync(p, s);
}

static std::atomic<long long> g_launches{0};
void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

int grid_1d(int64_t n)
{
    int64_t b = (n + 255) / 256;
    return (int)std::max<int64_t>(1, std::min<int64_t>(b, 152 * 32));
}

int bits_for(int64_t max_key)
{
    int b = 1;
    while (b < 32 && (max_key >> b) > 0) ++b;
    return b;
}

// ------------------------------------------------------------------ radix sort
// Stable LSD radix sort, reduce-then-scan per pass (no inter-tile waiting):
//   1. k_rs_hist:  digit counts of every 4096-pair tile, written tile-major
//      (in the conflict build's first pass also the id checks);
//   2. k_rs_chunk_sum / k_rs_chunk_scan / k_rs_chunk_down: the counts in
//      digit-major order become the global output offset of each (tile,
//      digit), computed hierarchically over chunks of 256 tiles;
//   3. k_rs_scatter: each tile ranks its pairs stably (one ballot per
//      digit bit, per-warp running counts, prefix over warps and digits), stages
//      them in shared memory in output order, and writes every digit's run
//      with consecutive threads.
// Digits are D = 8..10 bits, equal for all passes (27-bit ids: 3 passes of 9).
constexpr int RS_THREADS = 256;
constexpr int RS_IPT = 16;
constexpr int RS_TILE = RS_THREADS * RS_IPT;   // pairs per tile
constexpr int RS_CHUNK = 256;                  // tiles per scan chunk

// Per-tile digit counts.  In the first pass of the conflict build the same
// read of the ids also checks them: each must be below `range` (else
// PDB_ERANGE; range = 0: no check), and the DESC_SPREAD counters at
// `descents` (when not null) gain, together, the number of positions i >= 1
// with (int32) key[i-1] >= (int32) key[i].
template <int D>
__global__ __launch_bounds__(RS_THREADS) void k_rs_hist(const uint32_t *__restrict__ keys, int64_t n, int shift,
                                                         uint32_t *__restrict__ hist, uint32_t range, int *descents,
                                                         int *status)
{
    constexpr int RADIX = 1 << D;
    // one count per digit for the block: shared-memory atomics on one address
    // from different warps do not wait on each other, so per-warp copies would
    // only add their clearing and summing
    __shared__ uint32_t h[RADIX];
    __shared__ int s_desc;
    if (read_status(status)) return;
    for (int i = threadIdx.x; i < RADIX; i += RS_THREADS) h[i] = 0;
    if (threadIdx.x == 0) s_desc = 0;
    const int64_t tile0 = (int64_t)blockIdx.x * RS_TILE;
    const int ntile = (int)min64(RS_TILE, n - tile0);
    uint32_t k[RS_IPT];
#pragma unroll
    for (int i = 0; i < RS_IPT; ++i) {
        const int idx = i * RS_THREADS + threadIdx.x;
        k[i] = idx < ntile ? __ldcs(keys + tile0 + idx) : 0u;
    }
    bool bad = false;
    int desc = 0;
    if (range || descents) {
        // the key before element idx: the previous lane's, and for lane 0 a load
        // (it sits in another warp, or in the tile before)
        const int lane = threadIdx.x & 31;
#pragma unroll
        for (int i = 0; i < RS_IPT; ++i) {
            const int idx = i * RS_THREADS + threadIdx.x;
            uint32_t before = __shfl_up_sync(FULL, k[i], 1);
            if (lane == 0 && tile0 + idx > 0 && idx < ntile) before = keys[tile0 + idx - 1];
            if (idx < ntile) {
                bad |= range && k[i] >= range;
                if (descents && tile0 + idx > 0) desc += (int32_t)before >= (int32_t)k[i] ? 1 : 0;
            }
        }
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < RS_IPT; ++i)
        if (i * RS_THREADS + (int)threadIdx.x < ntile) atomicAdd(&h[(k[i] >> shift) & (RADIX - 1)], 1u);
    __syncthreads();
    for (int d = threadIdx.x; d < RADIX; d += RS_THREADS) hist[(int64_t)blockIdx.x * RADIX + d] = h[d];
    if (range || descents) {
        for (int off = 16; off >= 1; off >>= 1) desc += __shfl_xor_sync(FULL, desc, off);
        if ((threadIdx.x & 31) == 0 && desc) atomicAdd(&s_desc, desc);
        if (__any_sync(FULL, bad) && (threadIdx.x & 31) == 0) set_status(status, PDB_ERANGE);
        __syncthreads();
        // one add per block, spread over DESC_SPREAD counters (one address would serialize them)
        if (threadIdx.x == 0 && s_desc && descents) atomicAdd(descents + (blockIdx.x % DESC_SPREAD), s_desc);
    }
}

// column sums of the [tile][digit] counts over each chunk of RS_CHUNK tiles (RADIX threads)
__global__ void k_rs_chunk_sum(const uint32_t *__restrict__ hist, int64_t n_tiles, int radix,
                               uint32_t *__restrict__ csum, const int *status)
{
    if (read_status(status)) return;
    const int64_t t0 = (int64_t)blockIdx.x * RS_CHUNK, t1 = min64(n_tiles, t0 + RS_CHUNK);
    uint32_t s = 0;
    for (int64_t t = t0; t < t1; ++t) s += hist[t * radix + threadIdx.x];
    csum[(int64_t)blockIdx.x * radix + threadIdx.x] = s;
}

// one block of RADIX threads: cbase[chunk][d] = (pairs with a smaller digit)
// + (pairs with digit d in earlier chunks)
__global__ void k_rs_chunk_scan(const uint32_t *__restrict__ csum, int64_t n_chunks, int radix,
                                uint32_t *__restrict__ cbase, const int *status)
{
    __shared__ uint32_t wsum[32];
    if (read_status(status)) return;
    const int d = threadIdx.x, lane = d & 31, warp = d >> 5;
    uint32_t tot = 0;
    for (int64_t c = 0; c < n_chunks; ++c) tot += csum[c * radix + d];
    uint32_t x = tot;
    for (int off = 1; off < 32; off <<= 1) {
        uint32_t y = __shfl_up_sync(FULL, x, off);
        if (lane >= off) x += y;
    }
    if (lane == 31) wsum[warp] = x;
    __syncthreads();
    uint32_t run = x - tot;
    for (int w = 0; w < warp; ++w) run += wsum[w];
    for (int64_t c = 0; c < n_chunks; ++c) {
        const uint32_t v = csum[c * radix + d];
        cbase[c * radix + d] = run;
        run += v;
    }
}

// hist[tile][d] <- global output offset of digit d for that tile
__global__ void k_rs_chunk_down(uint32_t *__restrict__ hist, int64_t n_tiles, int radix,
                                const uint32_t *__restrict__ cbase, const int *status)
{
    if (read_status(status)) return;
    const int64_t t0 = (int64_t)blockIdx.x * RS_CHUNK, t1 = min64(n_tiles, t0 + RS_CHUNK);
    uint32_t run = cbase[(int64_t)blockIdx.x * radix + threadIdx.x];
    for (int64_t t = t0; t < t1; t += 16) {       // 16 loads in flight, then 16 stores
        uint32_t v[16];
#pragma unroll
        for (int u = 0; u < 16; ++u) v[u] = t + u < t1 ? hist[(t + u) * radix + threadIdx.x] : 0u;
#pragma unroll
        for (int u = 0; u < 16; ++u)
            if (t + u < t1) {
                hist[(t + u) * radix + threadIdx.x] = run;
                run += v[u];
            }
    }
}

template <int D>
__global__ __launch_bounds__(RS_THREADS, 3) void k_rs_scatter(const uint32_t *__restrict__ kin,
                                                               const int32_t *__restrict__ vin,
                                                               uint32_t *__restrict__ kout, int32_t *__restrict__ vout,
                                                               int64_t n, int shift, const uint32_t *__restrict__ offs,
                                                               const int *status)
{
    constexpr int RADIX = 1 << D;
    constexpr unsigned MASK = RADIX - 1;
    constexpr int PER = (RADIX + RS_THREADS - 1) / RS_THREADS;
    extern __shared__ uint32_t smem[];
    uint32_t *s_wcnt = smem;                       // [WARPS][RADIX]
    uint32_t *s_tpre = s_wcnt + WARPS * RADIX;     // [RADIX] tile counts, then tile-local offsets
    uint32_t *s_base = s_tpre + RADIX;             // [RADIX] global offset of each digit for this tile
    uint32_t *s_keys = s_base + RADIX;             // [RS_TILE]
    int32_t *s_vals = (int32_t *)(s_keys + RS_TILE);   // [RS_TILE] values in output order
    int32_t *s_vin = s_vals + RS_TILE;                  // [RS_TILE] values in input order
    __shared__ uint32_t s_wtot[WARPS];
    if (read_status(status)) return;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t tile0 = (int64_t)blockIdx.x * RS_TILE;
    const int ntile = (int)min64(RS_TILE, n - tile0);
    const uint32_t *tkin = kin + tile0;
    const int wbase = warp * (32 * RS_IPT);
    if (vin) {
        // the tile's values travel to shared memory asynchronously while the keys are ranked
        // (16-byte copies; the tile start is 16 KB aligned and vin is a 256-byte aligned buffer)
        const int full = ntile & ~3;
        for (int c = tid * 4; c < full; c += RS_THREADS * 4) {
            const unsigned dst = (unsigned)__cvta_generic_to_shared(s_vin + c);
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(vin + tile0 + c) : "memory");
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
        for (int c = full + tid; c < ntile; c += RS_THREADS) s_vin[c] = vin[tile0 + c];
    }
    uint32_t key[RS_IPT], pos[RS_IPT];
#pragma unroll
    for (int i = 0; i < RS_IPT; ++i) {          // all loads in flight before any ranking
        const int idx = wbase + i * 32 + lane;
        key[i] = idx < ntile ? __ldcs(tkin + idx) : 0u;
    }
    for (int i = tid; i < WARPS * RADIX; i += RS_THREADS) s_wcnt[i] = 0;
    for (int d = tid; d < RADIX; d += RS_THREADS) s_base[d] = offs[(int64_t)blockIdx.x * RADIX + d];
    __syncthreads();
    const unsigned lt = lanemask_lt();
    const bool full = ntile == RS_TILE;     // every tile but the last: no invalid lanes
    // 1. lanes holding the same digit, for all the thread's elements at once
    //    (one ballot per digit bit plus the valid bit, intersected; the
    //    ballots of different elements are independent, so they overlap):
    //    rank among the equal lanes, run length, leader flag
    uint32_t info[RS_IPT];
#pragma unroll
    for (int i = 0; i < RS_IPT; ++i) {
        const int idx = wbase + i * 32 + lane;
        const bool valid = idx < ntile;
        const unsigned d = valid ? ((key[i] >> shift) & MASK) : (unsigned)RADIX;
        unsigned peers = full ? FULL : __ballot_sync(FULL, valid);
        if (!valid) peers = ~peers;
#pragma unroll
        for (int b = 0; b < D; ++b) {
            const unsigned m = __ballot_sync(FULL, (d >> b) & 1u);
            peers &= ((d >> b) & 1u) ? m : ~m;
        }
        info[i] = d | (__popc(peers & lt) << 16) | (__popc(peers) << 24);
    }
    // 2. per-warp running count of each digit (the only serial part)
#pragma unroll
    for (int i = 0; i < RS_IPT; ++i) {
        const unsigned d = info[i] & 0xffffu;
        const unsigned rank = (info[i] >> 16) & 0xffu;
        const bool valid = d < (unsigned)RADIX;
        const unsigned cnt = valid ? s_wcnt[warp * RADIX + d] : 0u;
        pos[i] = cnt + rank;
        __syncwarp();
        if (valid && rank == 0) s_wcnt[warp * RADIX + d] = cnt + (info[i] >> 24);
        __syncwarp();
    }
    __syncthreads();
    // per digit: exclusive prefix over the warps and the tile count
    for (int d = tid; d < RADIX; d += RS_THREADS) {
        uint32_t run = 0;
#pragma unroll
        for (int w = 0; w < WARPS; ++w) {
            const uint32_t c = s_wcnt[w * RADIX + d];
            s_wcnt[w * RADIX + d] = run;
            run += c;
        }
        s_tpre[d] = run;
    }
    __syncthreads();
    // tile-local exclusive prefix of the digit counts
    {
        uint32_t local[PER], sum = 0;
#pragma unroll
        for (int q = 0; q < PER; ++q) {
            const int d = tid * PER + q;
            local[q] = d < RADIX ? s_tpre[d] : 0u;
            sum += local[q];
        }
        uint32_t x = sum;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const uint32_t y = __shfl_up_sync(FULL, x, off);
            if (lane >= off) x += y;
        }
        if (lane == 31) s_wtot[warp] = x;
        __syncthreads();
        uint32_t excl = x - sum;
#pragma unroll
        for (int w = 0; w < WARPS; ++w) excl += w < warp ? s_wtot[w] : 0u;
#pragma unroll
        for (int q = 0; q < PER; ++q) {
            const int d = tid * PER + q;
            if (d < RADIX) {
                s_tpre[d] = excl;
                s_base[d] -= excl;    // output index = s_base[d] + (tile-local index)
            }
            excl += local[q];
        }
    }
    if (vin) asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
#pragma unroll
    for (int i = 0; i < RS_IPT; ++i) {
        const int idx = wbase + i * 32 + lane;
        if (idx < ntile) {
            const unsigned d = (key[i] >> shift) & MASK;
            const uint32_t li = s_tpre[d] + s_wcnt[warp * RADIX + d] + pos[i];
            s_keys[li] = key[i];
            s_vals[li] = vin ? s_vin[idx] : (int32_t)(tile0 + idx);
        }
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < RS_IPT; ++i) {
        const int li = i * RS_THREADS + tid;
        if (li < ntile) {
            const uint32_t k = s_keys[li];
            const unsigned d = (k >> shift) & MASK;
            const uint32_t dest = s_base[d] + (uint32_t)li;
            kout[dest] = k;
            vout[dest] = s_vals[li];
        }
    }
}

template <int D>
int radix_passes(const uint32_t *keys_in, const int32_t *vals_in, uint32_t *keys_out, int32_t *vals_out,
                 uint32_t *keys_tmp, int32_t *vals_tmp, int64_t n, int passes, int shift0, const int *status,
                 cudaStream_t s, uint32_t range = 0, int *descents = nullptr)
{
    constexpr int RADIX = 1 << D;
    const size_t smem = sizeof(uint32_t) * ((size_t)(WARPS + 2) * RADIX + 3 * RS_TILE);
    // set once per device (any device past the table: every call)
    static std::atomic<bool> configured[64];
    int dev = 0;
    cudaGetDevice(&dev);
    const bool known = dev >= 0 && dev < 64;
    if (!known || !configured[dev].load(std::memory_order_acquire)) {
        if (cudaFuncSetAttribute(k_rs_scatter<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
            cudaSuccess)
            return PDB_ECUDA;
        if (known) configured[dev].store(true, std::memory_order_release);
    }
    const int64_t n_tiles = (n + RS_TILE - 1) / RS_TILE;
    const int64_t n_chunks = (n_tiles + RS_CHUNK - 1) / RS_CHUNK;
    uint32_t *hist = nullptr, *csum = nullptr, *cbase = nullptr;
    int rc = alloc((void **)&hist, sizeof(uint32_t) * RADIX * n_tiles, s);
    rc = rc ? rc : alloc((void **)&csum, sizeof(uint32_t) * RADIX * n_chunks, s);
    rc = rc ? rc : alloc((void **)&cbase, sizeof(uint32_t) * RADIX * n_chunks, s);
    if (rc == PDB_OK) {
        const uint32_t *kin = keys_in;
        const int32_t *vin = vals_in;
        for (int p = 0; p < passes; ++p) {
            const bool to_out = ((passes - 1 - p) % 2) == 0;   // the last pass lands in *_out
            uint32_t *ko = to_out ? keys_out : keys_tmp;
            int32_t *vo = to_out ? vals_out : vals_tmp;
            const int shift = shift0 + D * p;
            k_rs_hist<D><<<(unsigned)n_tiles, RS_THREADS, 0, s>>>(kin, n, shift, hist, p == 0 ? range : 0u,
                                                                  p == 0 ? descents : nullptr, const_cast<int *>(status));
            note_launch();
            k_rs_chunk_sum<<<(unsigned)n_chunks, RADIX, 0, s>>>(hist, n_tiles, RADIX, csum, status);
            note_launch();
            k_rs_chunk_scan<<<1, RADIX, 0, s>>>(csum, n_chunks, RADIX, cbase, status);
            note_launch();
            k_rs_chunk_down<<<(unsigned)n_chunks, RADIX, 0, s>>>(hist, n_tiles, RADIX, cbase, status);
            note_launch();
            k_rs_scatter<D><<<(unsigned)n_tiles, RS_THREADS, smem, s>>>(kin, vin, ko, vo, n, shift, hist, status);
            note_launch();
            kin = ko;
            vin = vo;
        }
    }
    release(hist, s);
    release(csum, s);
    release(cbase, s);
    if (rc != PDB_OK) return rc;
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

int radix_sort(const uint32_t *keys_in, const int32_t *vals_in, uint32_t *keys_out, int32_t *vals_out,
               uint32_t *keys_tmp, int32_t *vals_tmp, int64_t n, int key_bits, const int *status, cudaStream_t s,
               uint32_t range, int *descents)
{
    if (n <= 0) return PDB_OK;
    // equal digit widths of 8..10 bits: 27-bit ids take 3 passes of 9
    const int kb = std::max(1, std::min(key_bits, 32));
    const int passes = (kb + 9) / 10;
    const int d = std::max(8, (kb + passes - 1) / passes);
    if (d == 8)
        return radix_passes<8>(keys_in, vals_in, keys_out, vals_out, keys_tmp, vals_tmp, n, passes, 0, status, s,
                               range, descents);
    if (d == 9)
        return radix_passes<9>(keys_in, vals_in, keys_out, vals_out, keys_tmp, vals_tmp, n, passes, 0, status, s,
                               range, descents);
    return radix_passes<10>(keys_in, vals_in, keys_out, vals_out, keys_tmp, vals_tmp, n, passes, 0, status, s,
                            range, descents);
}

int radix_sort_bits(const uint32_t *keys_in, const int32_t *vals_in, uint32_t *keys_out, int32_t *vals_out,
                    uint32_t *keys_tmp, int32_t *vals_tmp, int64_t n, int lo_bit, int hi_bit, const int *status,
                    cudaStream_t s)
{
    if (n <= 0 || hi_bit <= lo_bit) return PDB_OK;
    const int kb = std::min(hi_bit, 32) - lo_bit;
    const int passes = (kb + 9) / 10;
    const int d = std::max(8, (kb + passes - 1) / passes);
    if (d == 8)
        return radix_passes<8>(keys_in, vals_in, keys_out, vals_out, keys_tmp, vals_tmp, n, passes, lo_bit, status, s);
    if (d == 9)
        return radix_passes<9>(keys_in, vals_in, keys_out, vals_out, keys_tmp, vals_tmp, n, passes, lo_bit, status, s);
    return radix_passes<10>(keys_in, vals_in, keys_out, vals_out, keys_tmp, vals_tmp, n, passes, lo_bit, status, s);
}

// ------------------------------------------------------------------ segment bounds
// ptr[b] = first index whose key is >= b, for b in 0..n_bins (keys sorted);
// four consecutive keys per thread and iteration
__global__ void k_segment_bounds(const uint32_t *__restrict__ keys, int64_t n, int64_t n_bins, const int *n_bins_dev,
                                 int64_t *__restrict__ ptr, const int *status)
{
    if (read_status(status)) return;
    const int64_t nb = n_bins_dev ? (int64_t)*n_bins_dev : n_bins;
    const bool vec = ((uintptr_t)keys & 15) == 0;
    const int64_t groups = (n + 3) >> 2;
    for (int64_t gi = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; gi < groups;
         gi += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i0 = gi << 2;
        int64_t k[5];
        k[0] = i0 == 0 ? -1 : (int64_t)keys[i0 - 1];
        if (vec && i0 + 4 <= n) {
            const uint4 k4 = __ldcs(reinterpret_cast<const uint4 *>(keys) + gi);
            k[1] = k4.x; k[2] = k4.y; k[3] = k4.z; k[4] = k4.w;
        } else {
#pragma unroll
            for (int e = 0; e < 4; ++e) k[e + 1] = i0 + e < n ? (int64_t)keys[i0 + e] : nb;
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int64_t i = i0 + e;
            if (i >= n) break;
            for (int64_t b = k[e] + 1; b <= k[e + 1] && b <= nb; ++b) ptr[b] = i;
            if (i == n - 1)
                for (int64_t b = k[e + 1] + 1; b <= nb; ++b) ptr[b] = n;
        }
    }
}

__global__ void k_fill_i64(int64_t *p, int64_t n_bins, const int *n_bins_dev, int64_t v)
{
    const int64_t nb = n_bins_dev ? (int64_t)*n_bins_dev : n_bins;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i <= nb; i += (int64_t)gridDim.x * blockDim.x)
        p[i] = v;
}

int segment_bounds(const uint32_t *sorted_keys, int64_t n, int64_t n_bins, const int *n_bins_dev, int64_t *ptr,
                   const int *status, cudaStream_t s)
{
    if (n == 0) {
        k_fill_i64<<<64, 256, 0, s>>>(ptr, n_bins, n_bins_dev, 0); note_launch();
    } else {
        int64_t blocks = std::min<int64_t>((n + 1023) / 1024, 65536);
        k_segment_bounds<<<(unsigned)blocks, 256, 0, s>>>(sorted_keys, n, n_bins, n_bins_dev, ptr, status); note_launch();
    }
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

}  // namespace pdb

extern "C" int64_t pdb_launch_count(void) { return (int64_t)pdb::g_launches.load(); }
