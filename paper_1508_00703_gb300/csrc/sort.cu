// Stable LSD radix sort of (uint32 key, int32 value) pairs and segment
// bounds of sorted keys, plus the small host helpers of libpdb.
//
// One pass per 8-bit digit.  A pass is: per-tile digit histogram (tiles of
// 4096 pairs), a scan of the [tile][digit] counts in digit-major order done
// hierarchically (chunk column sums, one-block scan of the chunk sums, chunk
// down-sweep), and a scatter in which each tile ranks its pairs stably
// (warp match on the digit, per-warp running counts, block prefix), stages
// them in shared memory in output order and writes each digit's run with
// consecutive threads.
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>

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
    return (uint64_t)(s * 1e9);
}

// Keep freed stream-ordered allocations in the device's default pool instead
// of returning them to the driver at every synchronization (done once per
// device; affects only cudaMallocAsync users of that pool).
static void keep_pool(int device)
{
    static bool done[64] = {};
    if (device < 0 || device >= 64 || done[device]) return;
    cudaMemPool_t pool;
    if (cudaDeviceGetDefaultMemPool(&pool, device) == cudaSuccess) {
        uint64_t keep = UINT64_MAX;
        cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &keep);
    }
    done[device] = true;
}

int alloc(void **p, size_t bytes, cudaStream_t s)
{
    *p = nullptr;
    int dev = 0;
    cudaGetDevice(&dev);
    keep_pool(dev);
    if (bytes == 0) bytes = 256;
    bytes = (bytes + 255) & ~(size_t)255;
    if (cudaMallocAsync(p, bytes, s) != cudaSuccess) {
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
constexpr int RS_THREADS = 256;
constexpr int RS_IPT = 16;
constexpr int RS_TILE = RS_THREADS * RS_IPT;   // 4096 pairs per tile
constexpr int RS_CHUNK = 256;                  // tiles per scan chunk

__global__ __launch_bounds__(RS_THREADS) void k_rs_hist(const uint32_t *__restrict__ keys, int64_t n, int shift,
                                                         uint32_t *__restrict__ hist, const int *status)
{
    if (read_status(status)) return;
    __shared__ uint32_t h[WARPS][256];
    for (int i = threadIdx.x; i < WARPS * 256; i += RS_THREADS) (&h[0][0])[i] = 0;
    __syncthreads();
    const int warp = threadIdx.x >> 5;
    const int64_t base = (int64_t)blockIdx.x * RS_TILE;
#pragma unroll 4
    for (int i = 0; i < RS_IPT; ++i) {
        int64_t idx = base + i * RS_THREADS + threadIdx.x;
        if (idx < n) atomicAdd(&h[warp][(keys[idx] >> shift) & 255u], 1u);
    }
    __syncthreads();
    uint32_t sum = 0;
#pragma unroll
    for (int w = 0; w < WARPS; ++w) sum += h[w][threadIdx.x];
    hist[(int64_t)blockIdx.x * 256 + threadIdx.x] = sum;
}

// column sums of the [tile][digit] counts over each chunk of RS_CHUNK tiles
__global__ __launch_bounds__(256) void k_rs_chunk_sum(const uint32_t *__restrict__ hist, int64_t n_tiles,
                                                      uint32_t *__restrict__ csum, const int *status)
{
    if (read_status(status)) return;
    int64_t t0 = (int64_t)blockIdx.x * RS_CHUNK;
    int64_t t1 = min64(n_tiles, t0 + RS_CHUNK);
    uint32_t s = 0;
    for (int64_t t = t0; t < t1; ++t) s += hist[t * 256 + threadIdx.x];
    csum[(int64_t)blockIdx.x * 256 + threadIdx.x] = s;
}

// one block: cbase[chunk][d] = (pairs with a smaller digit) + (pairs with
// digit d in earlier chunks)
__global__ __launch_bounds__(256) void k_rs_chunk_scan(const uint32_t *__restrict__ csum, int64_t n_chunks,
                                                       uint32_t *__restrict__ cbase, const int *status)
{
    if (read_status(status)) return;
    __shared__ uint32_t tot[256];
    const int d = threadIdx.x;
    uint32_t run = 0;
    for (int64_t c = 0; c < n_chunks; ++c) run += csum[c * 256 + d];
    tot[d] = run;
    __syncthreads();
    if (d == 0) {
        uint32_t acc = 0;
        for (int i = 0; i < 256; ++i) {
            uint32_t v = tot[i];
            tot[i] = acc;
            acc += v;
        }
    }
    __syncthreads();
    run = tot[d];
    for (int64_t c = 0; c < n_chunks; ++c) {
        uint32_t v = csum[c * 256 + d];
        cbase[c * 256 + d] = run;
        run += v;
    }
}

// hist[tile][d] <- global output offset of digit d for that tile
__global__ __launch_bounds__(256) void k_rs_chunk_down(uint32_t *__restrict__ hist, int64_t n_tiles,
                                                       const uint32_t *__restrict__ cbase, const int *status)
{
    if (read_status(status)) return;
    int64_t t0 = (int64_t)blockIdx.x * RS_CHUNK;
    int64_t t1 = min64(n_tiles, t0 + RS_CHUNK);
    uint32_t run = cbase[(int64_t)blockIdx.x * 256 + threadIdx.x];
    for (int64_t t = t0; t < t1; ++t) {
        uint32_t v = hist[t * 256 + threadIdx.x];
        hist[t * 256 + threadIdx.x] = run;
        run += v;
    }
}

__global__ __launch_bounds__(RS_THREADS) void k_rs_scatter(const uint32_t *__restrict__ kin,
                                                            const int32_t *__restrict__ vin,
                                                            uint32_t *__restrict__ kout, int32_t *__restrict__ vout,
                                                            int64_t n, int shift, const uint32_t *__restrict__ offs,
                                                            const int *status)
{
    if (read_status(status)) return;
    __shared__ uint32_t s_wcnt[WARPS][256];
    __shared__ uint32_t s_tpre[256];
    __shared__ uint32_t s_base[256];
    __shared__ uint32_t s_wtot[WARPS];
    __shared__ uint32_t s_keys[RS_TILE];
    __shared__ int32_t s_vals[RS_TILE];

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    for (int i = tid; i < WARPS * 256; i += RS_THREADS) (&s_wcnt[0][0])[i] = 0;
    s_base[tid] = offs[(int64_t)blockIdx.x * 256 + tid];
    __syncthreads();

    const int64_t tile0 = (int64_t)blockIdx.x * RS_TILE;
    const int64_t wbase = tile0 + (int64_t)warp * (32 * RS_IPT);
    const unsigned lt = lanemask_lt();
    uint32_t key[RS_IPT];
    int32_t val[RS_IPT];
    uint32_t pos[RS_IPT];
#pragma unroll
    for (int i = 0; i < RS_IPT; ++i) {
        int64_t idx = wbase + i * 32 + lane;
        bool valid = idx < n;
        key[i] = valid ? kin[idx] : 0u;
        val[i] = valid ? (vin ? vin[idx] : (int32_t)idx) : 0;
        unsigned d = valid ? ((key[i] >> shift) & 255u) : 256u;
        unsigned peers = __match_any_sync(FULL, d);
        unsigned rank = __popc(peers & lt);
        unsigned cnt = valid ? s_wcnt[warp][d] : 0u;
        pos[i] = cnt + rank;
        __syncwarp();
        if (valid && rank == 0) s_wcnt[warp][d] = cnt + __popc(peers);
        __syncwarp();
    }
    __syncthreads();
    // per digit: exclusive prefix over warps, then over digits for the tile
    {
        const int d = tid;
        uint32_t run = 0;
#pragma unroll
        for (int w = 0; w < WARPS; ++w) {
            uint32_t c = s_wcnt[w][d];
            s_wcnt[w][d] = run;
            run += c;
        }
        // block exclusive scan of run over d = 0..255
        uint32_t x = run;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            uint32_t y = __shfl_up_sync(FULL, x, off);
            if (lane >= off) x += y;
        }
        if (lane == 31) s_wtot[warp] = x;
        __syncthreads();
        uint32_t wpre = 0;
#pragma unroll
        for (int w = 0; w < WARPS; ++w) wpre += (w < warp) ? s_wtot[w] : 0u;
        s_tpre[d] = wpre + x - run;
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < RS_IPT; ++i) {
        int64_t idx = wbase + i * 32 + lane;
        if (idx < n) {
            unsigned d = (key[i] >> shift) & 255u;
            uint32_t li = s_tpre[d] + s_wcnt[warp][d] + pos[i];
            s_keys[li] = key[i];
            s_vals[li] = val[i];
        }
    }
    __syncthreads();
    const int64_t ntile = min64(RS_TILE, n - tile0);
#pragma unroll
    for (int i = 0; i < RS_IPT; ++i) {
        int li = i * RS_THREADS + tid;
        if (li < ntile) {
            uint32_t k = s_keys[li];
            unsigned d = (k >> shift) & 255u;
            uint32_t dest = s_base[d] + (uint32_t)li - s_tpre[d];
            kout[dest] = k;
            vout[dest] = s_vals[li];
        }
    }
}

int radix_sort(const uint32_t *keys_in, const int32_t *vals_in, uint32_t *keys_out, int32_t *vals_out,
               uint32_t *keys_tmp, int32_t *vals_tmp, int64_t n, int key_bits, const int *status, cudaStream_t s)
{
    if (n <= 0) return PDB_OK;
    const int passes = std::max(1, (key_bits + 7) / 8);
    const int64_t n_tiles = (n + RS_TILE - 1) / RS_TILE;
    const int64_t n_chunks = (n_tiles + RS_CHUNK - 1) / RS_CHUNK;
    uint32_t *hist = nullptr, *csum = nullptr, *cbase = nullptr;
    int rc = alloc((void **)&hist, sizeof(uint32_t) * 256 * n_tiles, s);
    if (rc == PDB_OK) rc = alloc((void **)&csum, sizeof(uint32_t) * 256 * n_chunks, s);
    if (rc == PDB_OK) rc = alloc((void **)&cbase, sizeof(uint32_t) * 256 * n_chunks, s);
    if (rc != PDB_OK) {
        release(hist, s);
        release(csum, s);
        release(cbase, s);
        return rc;
    }
    const uint32_t *kin = keys_in;
    const int32_t *vin = vals_in;
    for (int p = 0; p < passes; ++p) {
        // the last pass must land in *_out
        bool to_out = ((passes - 1 - p) % 2) == 0;
        uint32_t *ko = to_out ? keys_out : keys_tmp;
        int32_t *vo = to_out ? vals_out : vals_tmp;
        int shift = 8 * p;
        k_rs_hist<<<(unsigned)n_tiles, RS_THREADS, 0, s>>>(kin, n, shift, hist, status); note_launch();
        k_rs_chunk_sum<<<(unsigned)n_chunks, 256, 0, s>>>(hist, n_tiles, csum, status); note_launch();
        k_rs_chunk_scan<<<1, 256, 0, s>>>(csum, n_chunks, cbase, status); note_launch();
        k_rs_chunk_down<<<(unsigned)n_chunks, 256, 0, s>>>(hist, n_tiles, cbase, status); note_launch();
        k_rs_scatter<<<(unsigned)n_tiles, RS_THREADS, 0, s>>>(kin, vin, ko, vo, n, shift, hist, status); note_launch();
        kin = ko;
        vin = vo;
    }
    release(hist, s);
    release(csum, s);
    release(cbase, s);
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

// ------------------------------------------------------------------ segment bounds
__global__ void k_segment_bounds(const uint32_t *__restrict__ keys, int64_t n, int64_t n_bins, const int *n_bins_dev,
                                 int64_t *__restrict__ ptr, const int *status)
{
    if (read_status(status)) return;
    const int64_t nb = n_bins_dev ? (int64_t)*n_bins_dev : n_bins;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        int64_t k = keys[i];
        int64_t kp = i == 0 ? -1 : (int64_t)keys[i - 1];
        for (int64_t b = kp + 1; b <= k && b <= nb; ++b) ptr[b] = i;
        if (i == n - 1)
            for (int64_t b = k + 1; b <= nb; ++b) ptr[b] = n;
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
        int64_t blocks = std::min<int64_t>((n + 255) / 256, 65536);
        k_segment_bounds<<<(unsigned)blocks, 256, 0, s>>>(sorted_keys, n, n_bins, n_bins_dev, ptr, status); note_launch();
    }
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

}  // namespace pdb

extern "C" int64_t pdb_launch_count(void) { return (int64_t)pdb::g_launches.load(); }
