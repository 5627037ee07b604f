// Conflict structure and schedules: pdb_build_conflicts, pdb_schedule_build
// and the handle utilities of the C ABI.
//
// The read protocol of Section 5 keeps one iteration number per chunk and
// lets a read of iteration alpha+1 proceed once the chunk's number is alpha.
// With chunk = feature and iteration = example, that number becomes the
// per-feature occurrence rank, and the constraint links each occurrence to
// the previous occurrence of its feature: the chains built here.
//
// Layout: the (feature, position) pairs are stable-sorted by feature into
// csc_pos (one slot per nonzero, feature-major, data order inside a
// feature) delimited by feat_ptr.  Each position has one gate word: its
// occurrence rank (bits 0-28, the read protocol's iteration number), whether
// the next (bit 29) and the previous (bit 30) occurrence of its feature lie
// within `near` positions, and whether it is the feature's last occurrence
// (bit 31).  Up to 2^22 positions k_slots scatters the gate words straight
// to position order; above, the build keeps them in slot order (gate_sorted)
// plus the near pairs' words in position order (gate_window, all WINDOW
// needs), and ensure_gate builds the position-order array on first use.
// prev and next of a position follow from gate, feat_ptr and csc_pos by
// gathers and are materialized only when a caller asks for them.
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <atomic>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "common.cuh"

using namespace pdb;

namespace {

// device info words of a conflicts handle: status, longest chain, longest row,
// near occurrence pairs, and two descent counts (every position p >= 1 with
// col[p-1] >= col[p], and those where p starts a row: a row whose ids do not
// increase strictly is one with more of the first than of the second), each
// spread over DESC_SPREAD words
enum {
    INFO_STATUS = 0, INFO_MAX_CHAIN = 1, INFO_MAX_ROW = 2, INFO_NEAR = 4, INFO_DESC_ALL = 8,
    INFO_DESC_ROWS = INFO_DESC_ALL + DESC_SPREAD, INFO_WORDS = INFO_DESC_ROWS + DESC_SPREAD
};

// row_ptr[0] = 0, row_ptr[N] = nnz, nondecreasing (Definition 1: D is a list
// of examples); also the longest row and, for every row that is not empty and
// does not start the data, whether its first id is <= the id before it (the
// descents the feature sort counts over all positions, minus these, are the
// ones inside rows: only rows with one can repeat an id)
__global__ void k_validate_rows(const int64_t *__restrict__ row_ptr, const int32_t *__restrict__ col,
                                int64_t n_rows, int64_t nnz, int *info)
{
    int longest = 0, desc = 0;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t <= n_rows;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int64_t a = row_ptr[t];
        const int64_t e = t < n_rows ? row_ptr[t + 1] : a;
        const bool bad = (t == 0 && a != 0) || (t == n_rows && a != nnz) || e < a || a < 0 || a > nnz;
        if (bad) {
            set_status(info, PDB_EINVAL);
        } else if (t < n_rows && e <= nnz) {
            longest = max(longest, (int)(e - a));
            if (a > 0 && a < e) desc += col[a - 1] >= col[a] ? 1 : 0;
        }
    }
    __shared__ int s_longest, s_desc;
    if (threadIdx.x == 0) s_longest = s_desc = 0;
    __syncthreads();
    for (int off = 16; off >= 1; off >>= 1) {
        longest = max(longest, __shfl_xor_sync(FULL, longest, off));
        desc += __shfl_xor_sync(FULL, desc, off);
    }
    if ((threadIdx.x & 31) == 0) {
        if (longest > 0) atomicMax(&s_longest, longest);
        if (desc > 0) atomicAdd(&s_desc, desc);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        if (s_longest > 0) atomicMax(info + INFO_MAX_ROW, s_longest);
        if (s_desc > 0) atomicAdd(info + INFO_DESC_ROWS + blockIdx.x % DESC_SPREAD, s_desc);
    }
}

// example of each position (built on first use: LEVELS, CHAIN, BSP)
__global__ void k_row_of(const int64_t *__restrict__ row_ptr, int64_t n_rows, int32_t *__restrict__ row_of,
                         const int *info)
{
    if (read_status(info)) return;
    const int lane = threadIdx.x & 31;
    const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t t = gw; t < n_rows; t += nw) {
        const int64_t b = row_ptr[t], e = row_ptr[t + 1];
        for (int64_t p = b + lane; p < e; p += 32) row_of[p] = (int32_t)t;
    }
}

// the example holding position p: the last t with row_ptr[t] <= p
__device__ __forceinline__ int64_t find_row(const int64_t *__restrict__ row_ptr, int64_t n_rows, int64_t p)
{
    int64_t lo = 0, hi = n_rows - 1;
    while (lo < hi) {
        const int64_t mid = (lo + hi + 1) >> 1;
        if (row_ptr[mid] <= p)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

// The first slot of the run of key skey[q] (keys sorted): a gallop back from
// q, then a binary search in the last interval -- about 2 log2 of the run's
// length loads, once per warp
__device__ int64_t run_start(const uint32_t *__restrict__ skey, int64_t q)
{
    const uint32_t j = skey[q];
    int64_t hi = q, lo = q - 1, step = 1;          // skey[hi] == j
    while (lo >= 0 && skey[lo] == j) {
        hi = lo;
        step <<= 1;
        lo = hi - step;
    }
    if (lo < -1) lo = -1;                          // skey[lo] < j, or lo = -1
    while (hi - lo > 1) {
        const int64_t mid = lo + ((hi - lo) >> 1);
        if (skey[mid] == j)
            hi = mid;
        else
            lo = mid;
    }
    return hi;
}

// slots 4 gi .. 4 gi + 3 of the sorted keys and positions (0xffffffff and 0
// past the end); 16-byte loads where the group is whole
__device__ __forceinline__ void load_group(const uint32_t *__restrict__ skey, const int32_t *__restrict__ spos,
                                           int64_t nnz, int64_t gi, uint4 &k4, int4 &p4)
{
    const int64_t s0 = gi << 2;
    if (s0 + 4 <= nnz) {
        k4 = __ldcs(reinterpret_cast<const uint4 *>(skey) + gi);
        p4 = __ldcs(reinterpret_cast<const int4 *>(spos) + gi);
    } else {
        k4.x = s0 < nnz ? skey[s0] : 0xffffffffu;
        k4.y = s0 + 1 < nnz ? skey[s0 + 1] : 0xffffffffu;
        k4.z = s0 + 2 < nnz ? skey[s0 + 2] : 0xffffffffu;
        k4.w = s0 + 3 < nnz ? skey[s0 + 3] : 0xffffffffu;
        p4.x = s0 < nnz ? spos[s0] : 0;
        p4.y = s0 + 1 < nnz ? spos[s0 + 1] : 0;
        p4.z = s0 + 2 < nnz ? spos[s0 + 2] : 0;
        p4.w = s0 + 3 < nnz ? spos[s0 + 3] : 0;
    }
}

// Slot order: the gate word of every slot, rank | last-occurrence bit, the
// longest chain, feat_ptr (feat_ptr[b] = the first slot whose key is >= b,
// b = 0..n_cols) and -- only when some row is unsorted -- the repeated-id
// check: two neighbouring slots of one feature in the same example.  The
// gate words go to position order either directly (gate[csc_pos[s]], one
// scattered 4-byte store per slot) or, for large inputs, in slot order
// (gsort[s]) for the partitioned scatter below.
//
// Each warp takes a contiguous range of slots, 128 per step (four per lane,
// 16-byte loads and stores; the buffers come from the pool, 256-byte
// aligned), and carries the first slot of the run in progress from one step
// to the next, so a slot's rank is its distance to that slot without a
// second pass over the keys; the run in progress where the range begins is
// found once per warp by run_start.  feat_ptr is written per step, for the
// features from the key before the step to the step's last key, with
// consecutive features on consecutive lanes (stores that coalesce).
constexpr int SLOTS_THREADS = 256;

__global__ __launch_bounds__(SLOTS_THREADS) void k_slots(const uint32_t *__restrict__ skey,
                                                         const int32_t *__restrict__ spos, int64_t nnz, int64_t n_cols,
                                                         int64_t *__restrict__ feat_ptr,
                                                         const int64_t *__restrict__ row_ptr, int64_t n_rows,
                                                         int64_t near, uint32_t *__restrict__ gate,
                                                         uint32_t *__restrict__ gsort, uint32_t *__restrict__ gwin,
                                                         int *info)
{
    __shared__ bool s_check;
    __shared__ __align__(16) uint32_t s_keys[SLOTS_THREADS / 32][128];   // each warp's step of keys
    if (threadIdx.x == 0) {
        long long all = 0, rows = 0;
        for (int i = 0; i < DESC_SPREAD; ++i) {
            all += info[INFO_DESC_ALL + i];
            rows += info[INFO_DESC_ROWS + i];
        }
        s_check = all > rows;
    }
    __syncthreads();
    if (read_status(info)) return;
    const bool check_dup = s_check;
    const int lane = threadIdx.x & 31;
    uint32_t *sk = s_keys[threadIdx.x >> 5];
    const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t n_warps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int64_t steps = (nnz + 127) >> 7;
    const int64_t per = (steps + n_warps - 1) / n_warps;
    const int64_t st0 = warp * per, st1 = min(steps, st0 + per);
    int64_t carry = 0;                             // first slot of the run holding the slot before the step
    if (st0 < st1 && st0 > 0 && lane == 0) carry = run_start(skey, (st0 << 7) - 1);
    carry = __shfl_sync(FULL, carry, 0);
    // each step's keys and positions are loaded one step ahead, with the slot
    // after the step (lane 31); the slot before it is the last one of the step
    // before (lane 0), loaded only for the first step
    uint4 nk = make_uint4(0xffffffffu, 0xffffffffu, 0xffffffffu, 0xffffffffu);
    int4 np = make_int4(0, 0, 0, 0);
    uint32_t nke = 0xffffffffu, lk = 0xffffffffu;
    int32_t npe = 0, lp = 0;
    if (st0 < st1) {
        load_group(skey, spos, nnz, (st0 << 5) + lane, nk, np);
        const int64_t e = (st0 + 1) << 7;
        if (lane == 31 && e < nnz) {
            nke = skey[e];
            npe = spos[e];
        }
        if (lane == 0 && st0 > 0) {
            lk = skey[(st0 << 7) - 1];
            lp = spos[(st0 << 7) - 1];
        }
    }
    int longest = 0, n_near = 0;
    bool dup = false, big = false;
    for (int64_t st = st0; st < st1; ++st) {
        const int64_t gi = (st << 5) + lane;
        const int64_t s0 = gi << 2;
        uint32_t kk[6];
        int32_t pp[6];
        kk[1] = nk.x; kk[2] = nk.y; kk[3] = nk.z; kk[4] = nk.w;
        pp[1] = np.x; pp[2] = np.y; pp[3] = np.z; pp[4] = np.w;
        const uint32_t ke = nke;
        const int32_t pe = npe;
        if (st + 1 < st1) {
            load_group(skey, spos, nnz, gi + 32, nk, np);
            const int64_t e = (st + 2) << 7;
            nke = 0xffffffffu;
            npe = 0;
            if (lane == 31 && e < nnz) {
                nke = skey[e];
                npe = spos[e];
            }
        }
        // the neighbouring slots come from the lanes beside, the step's two
        // ends from the loads above (0xffffffff past either end of the keys)
        kk[0] = __shfl_up_sync(FULL, kk[4], 1);
        pp[0] = __shfl_up_sync(FULL, pp[4], 1);
        kk[5] = __shfl_down_sync(FULL, kk[1], 1);
        pp[5] = __shfl_down_sync(FULL, pp[1], 1);
        if (lane == 0) {
            kk[0] = lk;
            pp[0] = lp;
        }
        if (lane == 31) {
            kk[5] = ke;
            pp[5] = pe;
        }
        lk = __shfl_sync(FULL, kk[4], 31);
        lp = __shfl_sync(FULL, pp[4], 31);
        // the last run start among this lane's slots (offset in the step, -1
        // for none), its running maximum over the lanes, and from that the
        // first slot of the run that holds the slot before this lane's first
        int ls = -1;
#pragma unroll
        for (int e = 0; e < 4; ++e)
            if (s0 + e < nnz && kk[e] != kk[e + 1]) ls = lane * 4 + e;
        int inc = ls;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            const int t = __shfl_up_sync(FULL, inc, d);
            if (lane >= d) inc = max(inc, t);
        }
        int exc = __shfl_up_sync(FULL, inc, 1);
        if (lane == 0) exc = -1;
        const int64_t base = st << 7;
        const int64_t before = exc >= 0 ? base + exc : carry;
        const int last_start = __shfl_sync(FULL, inc, 31);
        if (last_start >= 0) carry = base + last_start;
        uint32_t g[4] = {0u, 0u, 0u, 0u};
        int64_t r = 0;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int64_t s = s0 + e;
            if (s >= nnz) break;
            const uint32_t j = kk[e + 1];
            const int32_t p = pp[e + 1];
            const bool first = kk[e] != j;
            const bool last = s == nnz - 1 || kk[e + 2] != j;
            // rank: 0 where the feature's run starts, one more than the slot
            // before inside the lane's slots, else the distance to the run's
            // first slot
            r = first ? 0 : e > 0 ? r + 1 : s - before;
            const bool near_prev = r > 0 && (int64_t)p - pp[e] < near;
            const bool near_next = !last && (int64_t)pp[e + 2] - p < near;
            big |= r > (int64_t)GATE_RANK;
            n_near += near_next;
            g[e] = ((uint32_t)r & GATE_RANK) | (near_next ? GATE_NEAR_NEXT : 0u) |
                   (near_prev ? GATE_NEAR_PREV : 0u) | (last ? GATE_LAST : 0u);
            if (!gsort) gate[p] = g[e];
            if (gwin && (near_prev || near_next)) gwin[p] = g[e];
            if (last) longest = max(longest, (int)(r + 1));
            if (check_dup && r > 0) dup |= find_row(row_ptr, n_rows, pp[e]) == find_row(row_ptr, n_rows, p);
        }
        if (gsort) {
            if (s0 + 4 <= nnz)
                __stcs(reinterpret_cast<uint4 *>(gsort) + gi, make_uint4(g[0], g[1], g[2], g[3]));
            else
                for (int e = 0; e < 4 && s0 + e < nnz; ++e) gsort[s0 + e] = g[e];
        }
        // feat_ptr[b] for the features b after the key before the step up to
        // the step's last key: the first slot of the step whose key is >= b
        // (a binary search in the step's keys), consecutive b on consecutive
        // lanes so that the stores coalesce; after the last slot of all, n
        *reinterpret_cast<uint4 *>(sk + lane * 4) = make_uint4(kk[1], kk[2], kk[3], kk[4]);
        __syncwarp();
        const int nv = (int)min((int64_t)128, nnz - base);
        const uint32_t kb = __shfl_sync(FULL, kk[0], 0);
        const int64_t khi = (int64_t)sk[nv - 1];
        const int64_t bhi = min(khi, n_cols);
        for (int64_t b = (base == 0 ? 0 : (int64_t)kb + 1) + lane; b <= bhi; b += 32) {
            int lo = 0, hi = nv;
            while (lo < hi) {
                const int mid = (lo + hi) >> 1;
                if ((int64_t)sk[mid] < b)
                    lo = mid + 1;
                else
                    hi = mid;
            }
            feat_ptr[b] = base + lo;
        }
        if (base + nv == nnz)
            for (int64_t b = khi + 1 + lane; b <= n_cols; b += 32) feat_ptr[b] = nnz;
        __syncwarp();                              // sk is rewritten by the next step
    }
    for (int off = 16; off >= 1; off >>= 1) {
        longest = max(longest, __shfl_xor_sync(FULL, longest, off));
        n_near += __shfl_xor_sync(FULL, n_near, off);
    }
    if (lane == 0 && longest > 0) atomicMax(info + INFO_MAX_CHAIN, longest);
    if (lane == 0 && n_near > 0) atomicAdd(info + INFO_NEAR, n_near);
    if (__any_sync(FULL, dup) && lane == 0) set_status(info, PDB_EDUP);
    if (__any_sync(FULL, big) && lane == 0) set_status(info, PDB_ETOOBIG);
}

// Last step of the gate scatter for large inputs.  The (position, gate)
// pairs arrive sorted on the position bits above SB, so block b of the pair
// array holds exactly the positions [b * 2^SB, (b + 1) * 2^SB) in some order
// (positions are a permutation of the slots).  One thread block inverts that
// piece in shared memory and writes it out contiguously: no ranking, and
// DRAM sees whole lines instead of one scattered 4-byte store per slot.
constexpr int SCATTER_SB = 14;                 // 2^14 slots = 64 KB of shared memory per block
constexpr int SCATTER_THREADS = 512;
__global__ __launch_bounds__(SCATTER_THREADS) void k_scatter_block(const uint32_t *__restrict__ ppos,
                                                                  const uint32_t *__restrict__ pgate, int64_t nnz,
                                                                  uint32_t *__restrict__ gate, int *info)
{
    extern __shared__ uint32_t piece[];
    if (read_status(info)) return;
    const int64_t base = (int64_t)blockIdx.x << SCATTER_SB;
    const int cnt = (int)min64((int64_t)1 << SCATTER_SB, nnz - base);
    bool bad = false;
    for (int i = threadIdx.x; i < cnt; i += SCATTER_THREADS) {
        const uint32_t off = __ldcs(ppos + base + i) - (uint32_t)base;
        if (off < (uint32_t)cnt)
            piece[off] = __ldcs(pgate + base + i);
        else
            bad = true;
    }
    if (bad) set_status(info, PDB_EFAULT);
    __syncthreads();
    for (int i = threadIdx.x; i < cnt; i += SCATTER_THREADS) gate[base + i] = piece[i];
}

// Position order: rank, previous and next occurrence of each position's feature.
__global__ void k_materialize(const int32_t *__restrict__ col, const uint32_t *__restrict__ gate,
                              const int32_t *__restrict__ csc_pos, const int64_t *__restrict__ feat_ptr, int64_t nnz,
                              int32_t *__restrict__ prev, int32_t *__restrict__ next, int32_t *__restrict__ rank,
                              const int *info)
{
    if (read_status(info)) return;
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < nnz; p += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t g = gate[p];
        const int32_t r = (int32_t)(g & GATE_RANK);
        const int64_t s = feat_ptr[col[p]] + r;
        rank[p] = r;
        prev[p] = r > 0 ? csc_pos[s - 1] : -1;
        next[p] = (g & GATE_LAST) ? -1 : csc_pos[s + 1];
    }
}

// per example: number of its positions whose feature occurred before (the
// in-degree of the example in the conflict DAG, counted per edge)
__global__ void k_npred(const int64_t *__restrict__ row_ptr, int64_t n_rows, const int32_t *__restrict__ prev,
                        int32_t *__restrict__ npred, const int *info)
{
    if (read_status(info)) return;
    const int lane = threadIdx.x & 31;
    const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t t = gw; t < n_rows; t += nw) {
        const int64_t b = row_ptr[t], e = row_ptr[t + 1];
        int cnt = 0;
        for (int64_t p = b + lane; p < e; p += 32) cnt += prev[p] >= 0;
        for (int off = 16; off >= 1; off >>= 1) cnt += __shfl_xor_sync(FULL, cnt, off);
        if (lane == 0) npred[t] = cnt;
    }
}

// append the flagged lanes' items to a global queue (one atomic per warp)
__device__ __forceinline__ int warp_append(bool flag, int *tail)
{
    unsigned m = __ballot_sync(FULL, flag);
    if (m == 0) return -1;
    const int lane = threadIdx.x & 31;
    const int leader = __ffs(m) - 1;
    int base = 0;
    if (lane == leader) base = atomicAdd(tail, __popc(m));
    base = __shfl_sync(FULL, base, leader);
    return flag ? base + __popc(m & lanemask_lt()) : -1;
}

// Kahn-style frontier sweep over the conflict DAG (edge: occurrence p ->
// next occurrence of the same feature).  Frontier l holds the examples all
// of whose predecessors are in frontiers < l; an example joins frontier l+1
// when its last incoming edge is consumed, which gives exactly the
// longest-path level.  One cooperative persistent launch; the frontiers are
// consecutive ranges of one queue, a grid barrier separates them, and the
// barrier's last arriver snapshots the queue end for everybody.
__global__ __launch_bounds__(THREADS) void k_levels_kahn(int32_t n_rows, const int64_t *__restrict__ row_ptr,
                                                         const int32_t *__restrict__ next,
                                                         const int32_t *__restrict__ row_of,
                                                         const int32_t *__restrict__ npred, int32_t *indeg,
                                                         int32_t *queue, int32_t *level, LevelCtl *ctl, int *status,
                                                         uint64_t timeout)
{
    if (read_status(status)) return;
    const int lane = threadIdx.x & 31;
    const int gw = (int)(((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
    const int nw = (int)(((int64_t)gridDim.x * blockDim.x) >> 5);
    for (int t0 = gw * 32; t0 < n_rows; t0 += nw * 32) {
        int t = t0 + lane;
        bool zero = false;
        if (t < n_rows) {
            int d = npred[t];
            indeg[t] = d;
            zero = d == 0;
            if (zero) level[t] = 0;
        }
        int slot = warp_append(zero, &ctl->tail);
        if (zero) queue[slot] = t;
    }
    if (!grid_sync(&ctl->bar, status, timeout, &ctl->tail, &ctl->end)) return;
    int head = 0, end = ld_acquire_i(&ctl->end), lvl = 0, widest = 0;
    while (head < end) {
        widest = max(widest, end - head);
        for (int i = head + gw; i < end; i += nw) {
            int t = __ldcg(queue + i);
            if (t < 0 || t >= n_rows) {        // cannot happen with a consistent queue
                set_status(status, PDB_EFAULT);
                continue;
            }
            int64_t b = row_ptr[t], e = row_ptr[t + 1];
            for (int64_t p0 = b; p0 < e; p0 += 32) {
                int64_t p = p0 + lane;
                bool fire = false;
                int u = -1;
                if (p < e) {
                    int q = next[p];
                    if (q >= 0) {
                        u = row_of[q];
                        fire = atomicSub(indeg + u, 1) == 1;
                    }
                }
                int slot = warp_append(fire, &ctl->tail);
                if (fire) {
                    queue[slot] = u;
                    level[u] = lvl + 1;
                }
            }
        }
        if (!grid_sync(&ctl->bar, status, timeout, &ctl->tail, &ctl->end)) return;
        head = end;
        end = ld_acquire_i(&ctl->end);
        ++lvl;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        ctl->n_levels = lvl;
        ctl->max_width = widest;
        if (end != n_rows) set_status(status, PDB_EFAULT);
    }
}

// Theorem 3's levels by dataflow instead of frontiers: warps take examples
// in data order from a ticket counter; example t waits (bounded) until the
// example of every previous occurrence of its features has published its
// level, then publishes 1 + their maximum (0 when there is none).  level[]
// starts at -1 (unpublished).  An example waits only on smaller ones and the
// smallest unfinished one on none, so there is no deadlock, and no grid
// barrier: a chain of L levels costs L hand-offs through L2, not L barriers.
__global__ __launch_bounds__(THREADS) void k_levels_flow(int32_t n_rows, const int64_t *__restrict__ row_ptr,
                                                         const int32_t *__restrict__ prev,
                                                         const int32_t *__restrict__ row_of, int32_t *level,
                                                         unsigned long long *ticket, int chunk, int *status,
                                                         uint64_t timeout)
{
    if (read_status(status)) return;
    const int lane = threadIdx.x & 31;
    for (;;) {
        unsigned long long tk = 0;
        if (lane == 0) tk = atomicAdd(ticket, (unsigned long long)chunk);
        tk = __shfl_sync(FULL, tk, 0);
        if (tk >= (unsigned long long)n_rows) return;
        const int t1 = (int)min64(n_rows, (int64_t)tk + chunk);
        for (int t = (int)tk; t < t1; ++t) {
            const int64_t b = row_ptr[t], e = row_ptr[t + 1];
            int best = -1;
            bool ok = true;
            for (int64_t p = b + lane; p < e && ok; p += 32) {
                const int q = prev[p];
                if (q < 0) continue;
                const int u = row_of[q];
                if (u < 0 || u >= t) {             // cannot happen with consistent chains
                    set_status(status, PDB_EFAULT);
                    ok = false;
                    break;
                }
                int lv = ld_acquire_i(level + u);
                if (lv < 0) {
                    const uint64_t t0 = globaltimer();
                    unsigned spins = 0, nap = 32;
                    while ((lv = ld_acquire_i(level + u)) < 0) {
                        __nanosleep(nap);
                        nap = nap < 256 ? 2 * nap : 256;
                        if ((++spins & 15u) != 0) continue;
                        if (read_status(status)) {
                            ok = false;
                            break;
                        }
                        if (globaltimer() - t0 > timeout) {
                            set_status(status, PDB_ETIMEOUT);
                            ok = false;
                            break;
                        }
                    }
                }
                best = max(best, lv);
            }
            if (!__all_sync(FULL, ok)) return;
            for (int off = 16; off >= 1; off >>= 1) best = max(best, __shfl_xor_sync(FULL, best, off));
            if (lane == 0) st_release(reinterpret_cast<unsigned *>(level + t), (unsigned)(best + 1));
        }
    }
}

// L = 1 + the largest level (the last of the sorted level keys)
__global__ void k_level_count(const uint32_t *__restrict__ sorted_levels, int32_t n, LevelCtl *ctl,
                              const int *status)
{
    if (read_status(status)) return;
    if (threadIdx.x == 0) ctl->n_levels = n > 0 ? (int)sorted_levels[n - 1] + 1 : 0;
}

// the widest level, from the level boundaries
__global__ void k_level_width(const int64_t *__restrict__ level_ptr, LevelCtl *ctl, const int *status)
{
    if (read_status(status)) return;
    const int L = ctl->n_levels;
    int widest = 0;
    for (int l = blockIdx.x * blockDim.x + threadIdx.x; l < L; l += gridDim.x * blockDim.x)
        widest = max(widest, (int)(level_ptr[l + 1] - level_ptr[l]));
    for (int off = 16; off >= 1; off >>= 1) widest = max(widest, __shfl_xor_sync(FULL, widest, off));
    if ((threadIdx.x & 31) == 0 && widest > 0) atomicMax(&ctl->max_width, widest);
}

__global__ void k_level_keys(const int32_t *__restrict__ level, uint32_t *__restrict__ key, int32_t n,
                             const int *status)
{
    if (read_status(status)) return;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) key[i] = (uint32_t)level[i];
}

int check_csr(const pdb_csr *X)
{
    if (!X || X->n_rows < 0 || X->n_cols < 0 || X->nnz < 0) return PDB_EINVAL;
    if (X->n_rows >= (1ll << 31) - 1 || X->n_cols >= (1ll << 31) - 1 || X->nnz >= (1ll << 31) - 1) return PDB_EINVAL;
    if (!X->row_ptr) return PDB_EINVAL;
    if (X->nnz > 0 && (!X->col || X->n_cols == 0)) return PDB_EINVAL;
    return PDB_OK;
}

// Callers wait for the handle's last use first (its ev_use), so the arrays
// are idle: they go back to the stream-ordered pool (kept, not returned to the
// driver) on the library's own stream, and the next allocation on any stream
// reuses them without an ordering against the legacy default stream (which
// would wait for every blocking stream's pending work).
void free_ptrs(std::initializer_list<void *> ptrs)
{
    cudaStream_t s = own_stream();
    for (void *p : ptrs)
        if (p) cudaFreeAsync(p, s);
}

}  // namespace

namespace pdb {

// row_of of every position (idempotent; enqueued on s)
int ensure_row_of(pdb_conflicts *c, cudaStream_t s)
{
    if (c->row_of) return PDB_OK;
    int32_t *row_of = nullptr;
    int rc = alloc((void **)&row_of, sizeof(int32_t) * std::max<int64_t>(c->nnz, 1), s);
    if (rc != PDB_OK) return rc;
    if (c->n_rows > 0) {
        k_row_of<<<grid_1d(c->n_rows * 32), 256, 0, s>>>(c->row_ptr, c->n_rows, row_of, c->status);
        note_launch();
    }
    c->row_of = row_of;
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

}  // namespace pdb

namespace {

// The position-order gate array (idempotent; enqueued on s).  Above 2^22
// positions the build keeps the gate words in csc_pos order only; here the
// (position, gate) pairs are sorted on the position bits above SCATTER_SB
// and k_scatter_block inverts each 2^SCATTER_SB-slot block in shared memory.
int ensure_gate(pdb_conflicts *c, cudaStream_t s)
{
    if (c->gate) return PDB_OK;
    const int64_t nnz = c->nnz;
    uint32_t *gate = nullptr, *pk = nullptr, *tkey = nullptr;
    int32_t *pv = nullptr, *tval = nullptr;
    int rc = alloc((void **)&gate, sizeof(uint32_t) * nnz, s);
    rc = rc ? rc : alloc((void **)&pk, sizeof(uint32_t) * nnz, s);
    rc = rc ? rc : alloc((void **)&pv, sizeof(int32_t) * nnz, s);
    rc = rc ? rc : alloc((void **)&tkey, sizeof(uint32_t) * nnz, s);
    rc = rc ? rc : alloc((void **)&tval, sizeof(int32_t) * nnz, s);
    if (rc == PDB_OK)
        rc = radix_sort_bits((const uint32_t *)c->csc_pos, (const int32_t *)c->gate_sorted, pk, pv, tkey, tval, nnz,
                             SCATTER_SB, bits_for(nnz - 1), c->info, s);
    if (rc == PDB_OK) {
        const size_t smem = sizeof(uint32_t) << SCATTER_SB;
        // set once per device (any device past the table: every call)
        static std::atomic<bool> configured[64];
        const bool known = c->device >= 0 && c->device < 64;
        if (!known || !configured[c->device].load(std::memory_order_acquire)) {
            if (cudaFuncSetAttribute(k_scatter_block, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
                cudaSuccess)
                rc = PDB_ECUDA;
            else if (known)
                configured[c->device].store(true, std::memory_order_release);
        }
        if (rc == PDB_OK) {
            const int64_t blocks = ((nnz - 1) >> SCATTER_SB) + 1;
            k_scatter_block<<<(unsigned)blocks, SCATTER_THREADS, smem, s>>>(pk, (const uint32_t *)pv, nnz, gate,
                                                                             c->info);
            note_launch();
        }
    }
    release(pk, s);
    release(pv, s);
    release(tkey, s);
    release(tval, s);
    if (rc != PDB_OK) {
        release(gate, s);
        return rc;
    }
    c->gate = gate;
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

// prev/next/rank of every position (idempotent; enqueued on s)
int materialize_chains(pdb_conflicts *c, cudaStream_t s)
{
    if (c->prev) return PDB_OK;
    const int rg = ensure_gate(c, s);
    if (rg != PDB_OK) return rg;
    const int64_t nnz = c->nnz;
    int32_t *prev = nullptr, *next = nullptr, *rank = nullptr;
    int rc = alloc((void **)&prev, sizeof(int32_t) * nnz, s);
    rc = rc ? rc : alloc((void **)&next, sizeof(int32_t) * nnz, s);
    rc = rc ? rc : alloc((void **)&rank, sizeof(int32_t) * nnz, s);
    if (rc != PDB_OK) {
        release(prev, s);
        release(next, s);
        release(rank, s);
        return rc;
    }
    if (nnz > 0) {
        k_materialize<<<grid_1d(nnz), 256, 0, s>>>(c->col, c->gate, c->csc_pos, c->feat_ptr, nnz, prev, next, rank,
                                                   c->status);
        note_launch();
    }
    c->prev = prev;
    c->next = next;
    c->rank = rank;
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

}  // namespace

// ------------------------------------------------------------------ C ABI
namespace pdb {

void mark_use(const pdb_conflicts *c, const pdb_schedule *h, cudaStream_t s)
{
    if (c && c->ev_use) cudaEventRecord(c->ev_use, s);
    if (h && h->ev_use) cudaEventRecord(h->ev_use, s);
}

// Small device-to-host reads of handle words go on the caller's stream, or,
// where the call has none, on the library's own stream (own_stream): a plain
// cudaMemcpy runs on the legacy default stream, which waits for every
// blocking stream of the device.  They are made by a one-block kernel that
// stores the words into mapped pinned host memory, not by a copy: a
// device-to-host copy of a few bytes queues behind whatever large copy the
// caller has in flight on the same copy engine (a training loop's weights
// going back to the host, say), and the read would wait for it.
__global__ void k_copy_words(const uint32_t *__restrict__ src, uint32_t *__restrict__ dst, int n)
{
    for (int i = threadIdx.x; i < n; i += blockDim.x) dst[i] = src[i];
}

__global__ void k_fill_words(uint32_t *__restrict__ p, uint32_t v, int64_t n)
{
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        p[i] = v;
}

int fill_words(void *p, uint32_t v, size_t bytes, cudaStream_t s)
{
    if (bytes % 4 != 0) return PDB_EINVAL;
    const int64_t n = (int64_t)(bytes / 4);
    if (n == 0) return PDB_OK;
    k_fill_words<<<grid_1d(n), 256, 0, s>>>((uint32_t *)p, v, n);
    note_launch();
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

static int copy_words_to_host(int *pinned, const void *src, size_t bytes, cudaStream_t s)
{
    int *dev = nullptr;
    if (bytes % 4 != 0 || cudaHostGetDevicePointer((void **)&dev, pinned, 0) != cudaSuccess) {
        cudaGetLastError();
        return PDB_ECUDA;
    }
    k_copy_words<<<1, 128, 0, s>>>((const uint32_t *)src, (uint32_t *)dev, (int)(bytes / 4));
    note_launch();
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

static int read_words(void *dst, const void *src, size_t bytes, cudaStream_t s)
{
    if (bytes > sizeof(int) * INFO_WORDS) return PDB_EINVAL;
    int *stage = info_slot_take();          // a pinned, mapped slot of the info slab
    if (!stage) return PDB_ENOMEM;
    int rc = copy_words_to_host(stage, src, bytes, s);
    if (rc == PDB_OK && cudaStreamSynchronize(s) != cudaSuccess) rc = PDB_ECUDA;
    if (rc == PDB_OK) std::memcpy(dst, stage, bytes);
    cudaGetLastError();
    info_slot_give(stage);
    return rc;
}

static int read_words(void *dst, const void *src, size_t bytes)
{
    return read_words(dst, src, bytes, own_stream());
}

static std::mutex g_slot_lock;
static std::vector<int *> g_free_slots;

int *info_slot_take()
{
    std::lock_guard<std::mutex> guard(g_slot_lock);
    if (g_free_slots.empty()) {
        constexpr int SLOTS = 64;
        int *slab = nullptr;
        if (cudaHostAlloc((void **)&slab, sizeof(int) * INFO_WORDS * SLOTS, cudaHostAllocMapped | cudaHostAllocPortable) !=
            cudaSuccess) {
            cudaGetLastError();
            return nullptr;
        }
        for (int i = SLOTS - 1; i >= 0; --i) g_free_slots.push_back(slab + i * INFO_WORDS);
    }
    int *slot = g_free_slots.back();
    g_free_slots.pop_back();
    std::memset(slot, 0, sizeof(int) * INFO_WORDS);
    return slot;
}

void info_slot_give(int *slot)
{
    if (!slot) return;
    std::lock_guard<std::mutex> guard(g_slot_lock);
    g_free_slots.push_back(slot);
}

ApiScope::ApiScope(const char *name_, const pdb_conflicts *c_, const pdb_schedule *h_, pdb_conflicts *const *pc_,
                   pdb_schedule *const *ph_, bool log_)
    : name(name_), c(c_), h(h_), pc(pc_), ph(ph_), log(log_)
{
    nvtxRangePushA(name);
}

ApiScope::~ApiScope()
{
    nvtxRangePop();
    const char *env = std::getenv("PDB_LOG");
    if (!log || !env || !*env || std::strcmp(env, "0") == 0) return;
    const pdb_conflicts *cc = pc ? *pc : c;
    const pdb_schedule *hh = ph ? *ph : h;
    if (!cc && hh) cc = hh->c;
    pdb_stats st;
    if (!cc || pdb_get_stats(cc, hh, &st) != PDB_OK) {
        std::fprintf(stderr, "pdb %s: no handle\n", name);
        return;
    }
    int status = 0;
    read_words(&status, cc->status, sizeof status);
    std::fprintf(stderr,
                 "pdb %s: n_rows=%lld n_cols=%lld nnz=%lld max_chain=%lld sched_mode=%lld n_levels=%lld "
                 "max_level_width=%lld ms_build=%.3f ms_schedule=%.3f ms_sgd=%.3f ms_sgd_kernels=%.3f ms_bsp=%.3f "
                 "status=%d launches=%lld\n",
                 name, (long long)st.n_rows, (long long)st.n_cols, (long long)st.nnz, (long long)st.max_chain,
                 (long long)st.sched_mode, (long long)st.n_levels, (long long)st.max_level_width, st.ms_build,
                 st.ms_schedule, st.ms_sgd, st.ms_sgd_kernels, st.ms_bsp, status, (long long)pdb_launch_count());
}

}  // namespace pdb

extern "C" {

const char *pdb_strerror(int code)
{
    switch (code) {
    case PDB_OK: return "ok";
    case PDB_EINVAL: return "invalid argument or malformed row_ptr";
    case PDB_ERANGE: return "feature id outside [0, n_cols)";
    case PDB_EDUP: return "feature id repeated inside one example";
    case PDB_ENOMEM: return "device allocation failed";
    case PDB_ECUDA: return "CUDA runtime error";
    case PDB_ETIMEOUT: return "device-side wait expired";
    case PDB_EFAULT: return "internal invariant failed on the device";
    case PDB_ESTATE: return "handle in the wrong mode for this call";
    case PDB_ETOOBIG:
        return "problem beyond a fixed limit (allocation-free scratch: 2^20 features; CHAIN: 256 ids per example "
               "unless the weights fit in shared memory; a feature in 2^29 positions or more)";
    default: return "unknown error";
    }
}

void pdb_conflicts_free(pdb_conflicts *c)
{
    if (!c) return;
    // the handle's own work only: other streams of the device keep running
    if (c->ev_use) cudaEventSynchronize(c->ev_use);
    free_ptrs({c->csc_pos, c->feat_ptr, c->gate, c->gate_sorted, c->gate_window != c->gate ? c->gate_window : nullptr,
               c->row_of, c->prev, c->next, c->rank, c->npred, c->info});
    info_slot_give(c->h_info);
    for (cudaEvent_t e : {c->ev0, c->ev1, c->ev_sgd0, c->ev_sgd1, c->ev_bsp0, c->ev_bsp1, c->ev_k0, c->ev_k1, c->ev_use})
        if (e) cudaEventDestroy(e);
    delete c;
}

int pdb_build_conflicts(const pdb_csr *X, pdb_conflicts **out, void *stream)
{
    ApiScope scope("pdb_build_conflicts", nullptr, nullptr, out);
    if (!out) return PDB_EINVAL;
    *out = nullptr;
    int rc = check_csr(X);
    if (rc != PDB_OK) return rc;
    cudaStream_t s = (cudaStream_t)stream;
    pdb_conflicts *c = new (std::nothrow) pdb_conflicts();
    if (!c) return PDB_ENOMEM;
    cudaGetDevice(&c->device);
    c->n_rows = X->n_rows;
    c->n_cols = X->n_cols;
    c->nnz = X->nnz;
    c->row_ptr = X->row_ptr;
    c->col = X->col;
    c->val = X->val;
    const int64_t N = X->n_rows, F = X->n_cols, nnz = X->nnz;
    // WINDOW distance: several times the positions one persistent grid holds
    // in flight (~15k examples), at least 2^22
    {
        const int64_t k_mean = N > 0 ? (nnz + N - 1) / N : 1;
        int64_t near = (int64_t)1 << 22;
        while (near < k_mean * ((int64_t)1 << 15) && near < ((int64_t)1 << 29)) near <<= 1;
        // PDB_NEAR overrides it (any value >= 1 gives the same result; small
        // values exercise the watermark path on small inputs)
        if (const char *env = std::getenv("PDB_NEAR")) {
            const long long v = std::atoll(env);
            if (v >= 1) near = std::min<int64_t>(v, (int64_t)1 << 30);
        }
        c->near = near;
    }
    for (cudaEvent_t *e : {&c->ev0, &c->ev1, &c->ev_sgd0, &c->ev_sgd1, &c->ev_bsp0, &c->ev_bsp1, &c->ev_k0, &c->ev_k1})
        if (cudaEventCreate(e) != cudaSuccess) {
            pdb_conflicts_free(c);
            return PDB_ECUDA;
        }
    if (cudaEventCreateWithFlags(&c->ev_use, cudaEventDisableTiming) != cudaSuccess) {
        pdb_conflicts_free(c);
        return PDB_ECUDA;
    }
    c->h_info = info_slot_take();
    if (!c->h_info) {
        pdb_conflicts_free(c);
        return PDB_ENOMEM;
    }
    cudaEventRecord(c->ev0, s);
    rc = alloc((void **)&c->info, sizeof(int) * INFO_WORDS, s);
    rc = rc ? rc : alloc((void **)&c->csc_pos, sizeof(int32_t) * nnz, s);
    // up to 2^22 slots the gate array (16 MB) stays in L2 and k_slots scatters
    // it to position order directly; above, the build keeps it in slot order
    // plus a WINDOW gate holding only the near pairs' words, and the full
    // position-order array is built on first use (ensure_gate)
    const bool partition = nnz > 0 && bits_for(nnz - 1) > 22;
    if (!partition) {
        rc = rc ? rc : alloc((void **)&c->gate, sizeof(uint32_t) * std::max<int64_t>(nnz, 1), s);
        c->gate_window = c->gate;
    } else {
        rc = rc ? rc : alloc((void **)&c->gate_sorted, sizeof(uint32_t) * nnz, s);
        rc = rc ? rc : alloc((void **)&c->gate_window, sizeof(uint32_t) * nnz, s);
        if (rc == PDB_OK) rc = fill_words(c->gate_window, 0u, sizeof(uint32_t) * nnz, s);
    }
    rc = rc ? rc : alloc((void **)&c->feat_ptr, sizeof(int64_t) * (F + 1), s);
    uint32_t *skey = nullptr, *tkey = nullptr;
    int32_t *tval = nullptr;
    rc = rc ? rc : alloc((void **)&skey, sizeof(uint32_t) * nnz, s);
    rc = rc ? rc : alloc((void **)&tkey, sizeof(uint32_t) * nnz, s);
    rc = rc ? rc : alloc((void **)&tval, sizeof(int32_t) * nnz, s);
    c->status = c->info;
    if (rc == PDB_OK) {
        rc = fill_words(c->info, 0u, sizeof(int) * INFO_WORDS, s);
        k_validate_rows<<<grid_1d(N + 1), 256, 0, s>>>(X->row_ptr, X->col, N, nnz, c->info);
        note_launch();
        // (feature, position) pairs sorted by feature, stable: positions stay in data order.
        // The sort's first read of the ids also checks that they lie in [0, n_cols)
        // (PDB_ERANGE) and counts the descents.
        rc = rc ? rc : radix_sort((const uint32_t *)X->col, nullptr, skey, c->csc_pos, tkey, tval, nnz,
                        bits_for(F > 0 ? F - 1 : 0), c->info, s, (uint32_t)F, c->info + INFO_DESC_ALL);
    }
    // k_slots writes feat_ptr; with no nonzeros every bound is 0
    if (rc == PDB_OK && nnz == 0) rc = segment_bounds(skey, 0, F, nullptr, c->feat_ptr, c->info, s);
    if (rc == PDB_OK && nnz > 0) {
        k_slots<<<grid_1d((nnz + 3) / 4), SLOTS_THREADS, 0, s>>>(skey, c->csc_pos, nnz, F, c->feat_ptr, X->row_ptr, N,
                                                        c->near, c->gate, c->gate_sorted,
                                                        partition ? c->gate_window : nullptr, c->info);
        note_launch();
    }
    release(skey, s);
    release(tkey, s);
    release(tval, s);
    if (rc == PDB_OK) rc = copy_words_to_host(c->h_info, c->info, sizeof(int) * INFO_WORDS, s);
    cudaEventRecord(c->ev1, s);
    mark_use(c, nullptr, s);
    c->timed_build = true;
    if (rc == PDB_OK && cudaPeekAtLastError() != cudaSuccess) rc = PDB_ECUDA;
    if (rc != PDB_OK) {
        cudaGetLastError();
        cudaStreamSynchronize(s);
        pdb_conflicts_free(c);
        return rc;
    }
    *out = c;
    return PDB_OK;
}

int pdb_conflicts_arrays(const pdb_conflicts *c, const int32_t **csc_pos, const int64_t **feat_ptr,
                         const int32_t **prev, const int32_t **next, const int32_t **rank, void *stream)
{
    if (!c) return PDB_EINVAL;
    pdb_conflicts *cm = const_cast<pdb_conflicts *>(c);
    if (prev || next || rank) {
        int rc = materialize_chains(cm, (cudaStream_t)stream);
        mark_use(c, nullptr, (cudaStream_t)stream);
        if (rc != PDB_OK) return rc;
    }
    if (csc_pos) *csc_pos = c->csc_pos;
    if (feat_ptr) *feat_ptr = c->feat_ptr;
    if (prev) *prev = c->prev;
    if (next) *next = c->next;
    if (rank) *rank = c->rank;
    return PDB_OK;
}

int pdb_status(const pdb_conflicts *c, void *stream)
{
    if (!c) return PDB_EINVAL;
    int st = 0;
    if (read_words(&st, c->status, sizeof(int), (cudaStream_t)stream) != PDB_OK) return PDB_ECUDA;   // after the stream's work
    return st;
}

void pdb_schedule_free(pdb_schedule *s)
{
    if (!s) return;
    // the schedule's own work only: other streams of the device keep running
    if (s->ev_use) cudaEventSynchronize(s->ev_use);
    free_ptrs({s->level, s->order, s->indeg, s->queue, s->level_ptr, s->ctl, s->rec, s->link, s->bar, s->ticket,
               s->prog, s->wctl, s->reads, s->writes, s->rbits, s->wbits});
    for (cudaEvent_t e : {s->ev0, s->ev1, s->ev_use})
        if (e) cudaEventDestroy(e);
    delete s;
}

int pdb_schedule_build(const pdb_conflicts *c, pdb_sched_mode mode, pdb_schedule **out, void *stream)
{
    ApiScope scope("pdb_schedule_build", c, nullptr, nullptr, out);
    if (!c || !out || mode < PDB_SCHED_LEVELS || mode > PDB_SCHED_WINDOW) return PDB_EINVAL;
    *out = nullptr;
    cudaStream_t s = (cudaStream_t)stream;
    pdb_conflicts *cm = const_cast<pdb_conflicts *>(c);
    if (mode == PDB_SCHED_CHAIN || mode == PDB_SCHED_AUTO) {
        // both need the longest row (and AUTO the longest chain) recorded by the build
        if (cudaEventSynchronize(c->ev1) != cudaSuccess) {
            cudaGetLastError();
            return PDB_ECUDA;
        }
        const bool fits = c->h_info[INFO_MAX_ROW] <= chain_max_row() ||
                          resident_smem(c->n_cols, c->h_info[INFO_MAX_ROW]) > 0;
        // AUTO: one chain dominates -> CHAIN; near occurrence pairs rare
        // (at most 1/8 of the positions) -> WINDOW; else READY
        if (mode == PDB_SCHED_AUTO)
            mode = (fits && (int64_t)c->h_info[INFO_MAX_CHAIN] * 20 > c->n_rows) ? PDB_SCHED_CHAIN
                   : (int64_t)c->h_info[INFO_NEAR] * 8 <= c->nnz                  ? PDB_SCHED_WINDOW
                                                                                 : PDB_SCHED_READY;
        else if (!fits)
            return PDB_ETOOBIG;
    }
    pdb_schedule *h = new (std::nothrow) pdb_schedule();
    if (!h) return PDB_ENOMEM;
    h->c = c;
    h->mode = mode;
    if (cudaEventCreate(&h->ev0) != cudaSuccess || cudaEventCreate(&h->ev1) != cudaSuccess ||
        cudaEventCreateWithFlags(&h->ev_use, cudaEventDisableTiming) != cudaSuccess) {
        pdb_schedule_free(h);
        return PDB_ECUDA;
    }
    const int64_t N = c->n_rows, F = c->n_cols, nnz = c->nnz;
    cudaEventRecord(h->ev0, s);
    int rc = alloc((void **)&h->bar, sizeof(GridBarrier), s);
    rc = rc ? rc : alloc((void **)&h->ticket, sizeof(unsigned long long), s);
    if (rc == PDB_OK) {
        rc = fill_words(h->bar, 0u, sizeof(GridBarrier), s);
        rc = rc ? rc : fill_words(h->ticket, 0u, sizeof(unsigned long long), s);
    }
    if (mode == PDB_SCHED_READY) {
        // one (weight, version) record per feature; filled from w by pdb_sgd_epoch;
        // every position's gate word
        rc = rc ? rc : ensure_gate(cm, s);
        rc = rc ? rc : alloc((void **)&h->rec, sizeof(unsigned long long) * F, s);
    } else if (mode == PDB_SCHED_WINDOW) {
        // near hand-off records (tag 0 = none: tags carry a nonzero epoch
        // stamp), a done flag per chunk of examples (zeroed once: flags
        // carry the epoch's tag), the ticket and the watermark (reset every
        // epoch)
        h->prog_cap = (std::max<int64_t>(N, 1) + 3) & ~(int64_t)3;   // the sweeper reads four flags at a time
        rc = rc ? rc : alloc((void **)&h->rec, sizeof(unsigned long long) * std::max<int64_t>(F, 1), s);
        if (rc == PDB_OK) rc = fill_words(h->rec, 0u, sizeof(unsigned long long) * std::max<int64_t>(F, 1), s);
        rc = rc ? rc : alloc((void **)&h->prog, sizeof(unsigned) * h->prog_cap, s);
        if (rc == PDB_OK) rc = fill_words(h->prog, 0u, sizeof(unsigned) * h->prog_cap, s);
        rc = rc ? rc : alloc((void **)&h->wctl, sizeof(WindowCtl), s);
    } else if (mode == PDB_SCHED_CHAIN) {
        // rows longer than the forwarding engine takes: weights resident in
        // shared memory (they fit, checked above), no link words
        h->resident = c->h_info[INFO_MAX_ROW] > chain_max_row();
        if (!h->resident) {
            rc = rc ? rc : materialize_chains(cm, s);
            rc = rc ? rc : alloc((void **)&h->link, sizeof(uint32_t) * nnz, s);
            rc = rc ? rc : ensure_row_of(cm, s);
            rc = rc ? rc : chain_schedule(c->prev, c->next, c->row_of, c->row_ptr, nnz, c->h_info[INFO_MAX_ROW], h->link,
                                          c->status, s);
        }
    } else {
        // Theorem 3's levels by dataflow (default) or by the Kahn frontier sweep
        // (PDB_LEVELS=kahn: one grid barrier per level)
        const char *lv_env = std::getenv("PDB_LEVELS");
        const bool flow = !(lv_env && std::strcmp(lv_env, "kahn") == 0);
        rc = rc ? rc : materialize_chains(cm, s);
        rc = rc ? rc : ensure_row_of(cm, s);
        if (!flow && rc == PDB_OK && !cm->npred) {
            rc = alloc((void **)&cm->npred, sizeof(int32_t) * N, s);
            if (rc == PDB_OK && N > 0) {
                k_npred<<<grid_1d(N * 32), 256, 0, s>>>(c->row_ptr, N, c->prev, cm->npred, c->status);
                note_launch();
            }
        }
        rc = rc ? rc : alloc((void **)&h->level, sizeof(int32_t) * N, s);
        rc = rc ? rc : alloc((void **)&h->order, sizeof(int32_t) * N, s);
        if (!flow) {
            rc = rc ? rc : alloc((void **)&h->indeg, sizeof(int32_t) * N, s);
            rc = rc ? rc : alloc((void **)&h->queue, sizeof(int32_t) * N, s);
        }
        rc = rc ? rc : alloc((void **)&h->level_ptr, sizeof(int64_t) * (N + 1), s);
        rc = rc ? rc : alloc((void **)&h->ctl, sizeof(LevelCtl), s);
        uint32_t *key = nullptr, *skey = nullptr, *tkey = nullptr;
        int32_t *tval = nullptr;
        rc = rc ? rc : alloc((void **)&key, sizeof(uint32_t) * N, s);
        rc = rc ? rc : alloc((void **)&skey, sizeof(uint32_t) * N, s);
        rc = rc ? rc : alloc((void **)&tkey, sizeof(uint32_t) * N, s);
        rc = rc ? rc : alloc((void **)&tval, sizeof(int32_t) * N, s);
        if (rc == PDB_OK) {
            rc = rc ? rc : fill_words(h->ctl, 0u, sizeof(LevelCtl), s);
            if (N > 0) {
                int32_t n32 = (int32_t)N;
                uint64_t tmo = timeout_ns(nullptr);
                if (flow) {
                    rc = fill_words(h->level, 0xffffffffu, sizeof(int32_t) * N, s);
                    rc = rc ? rc : fill_words(h->ticket, 0u, sizeof(unsigned long long), s);
                    const int grid = persistent_grid((const void *)k_levels_flow, nullptr);
                    k_levels_flow<<<grid, THREADS, 0, s>>>(n32, c->row_ptr, c->prev, c->row_of, h->level, h->ticket, 4,
                                                           c->status, tmo);
                    note_launch();
                } else {
                    const void *kern = (const void *)k_levels_kahn;
                    int grid = persistent_grid(kern, nullptr);
                    void *args[] = {&n32,       (void *)&c->row_ptr, (void *)&c->next, (void *)&c->row_of,
                                    (void *)&c->npred, &h->indeg, &h->queue, &h->level,
                                    &h->ctl,    (void *)&c->status, &tmo};
                    if (cudaLaunchCooperativeKernel(kern, grid, THREADS, args, 0, s) != cudaSuccess) rc = PDB_ECUDA;
                    note_launch();
                }
                if (rc == PDB_OK) {
                    k_level_keys<<<grid_1d(N), 256, 0, s>>>(h->level, key, n32, c->status);
                    note_launch();
                    rc = radix_sort(key, nullptr, skey, h->order, tkey, tval, N, bits_for(N), c->status, s);
                }
                if (rc == PDB_OK && flow) {
                    k_level_count<<<1, 32, 0, s>>>(skey, n32, h->ctl, c->status);
                    note_launch();
                }
                if (rc == PDB_OK) rc = segment_bounds(skey, N, N, &h->ctl->n_levels, h->level_ptr, c->status, s);
                if (rc == PDB_OK && flow) {
                    k_level_width<<<grid_1d(N), 256, 0, s>>>(h->level_ptr, h->ctl, c->status);
                    note_launch();
                }
            } else {
                rc = rc ? rc : fill_words(h->level_ptr, 0u, sizeof(int64_t), s);
            }
        }
        release(key, s);
        release(skey, s);
        release(tkey, s);
        release(tval, s);
    }
    cudaEventRecord(h->ev1, s);
    mark_use(c, h, s);     // the schedule's build also reads and extends c's arrays
    h->timed = true;
    if (rc == PDB_OK && cudaPeekAtLastError() != cudaSuccess) rc = PDB_ECUDA;
    if (rc != PDB_OK) {
        cudaGetLastError();
        cudaStreamSynchronize(s);
        pdb_schedule_free(h);
        return rc;
    }
    *out = h;
    return PDB_OK;
}

int pdb_schedule_levels(const pdb_schedule *h, const int32_t **level, const int32_t **order,
                        const int64_t **level_ptr, int64_t *n_levels, void *stream)
{
    if (!h) return PDB_EINVAL;
    if (h->mode != PDB_SCHED_LEVELS) return PDB_ESTATE;
    if (level) *level = h->level;
    if (order) *order = h->order;
    if (level_ptr) *level_ptr = h->level_ptr;
    if (n_levels) {
        LevelCtl ctl;
        if (read_words(&ctl, h->ctl, sizeof ctl, (cudaStream_t)stream) != PDB_OK) return PDB_ECUDA;
        *n_levels = h->c->n_rows > 0 ? ctl.n_levels : 0;
    }
    return PDB_OK;
}

int pdb_schedule_ready(const pdb_schedule *h, const uint32_t **gate, const uint64_t **records)
{
    if (!h) return PDB_EINVAL;
    if (h->mode != PDB_SCHED_READY && h->mode != PDB_SCHED_WINDOW) return PDB_ESTATE;
    if (gate) *gate = h->mode == PDB_SCHED_WINDOW ? h->c->gate_window : h->c->gate;
    if (records) *records = (const uint64_t *)h->rec;   // NULL under WINDOW
    return PDB_OK;
}

int pdb_get_stats(const pdb_conflicts *c, const pdb_schedule *h, pdb_stats *out)
{
    if (!c || !out) return PDB_EINVAL;
    std::memset(out, 0, sizeof *out);
    // the work enqueued on these handles (their timers and words are final then)
    if ((c->ev_use && cudaEventSynchronize(c->ev_use) != cudaSuccess) ||
        (h && h->ev_use && cudaEventSynchronize(h->ev_use) != cudaSuccess))
        return PDB_ECUDA;
    out->n_rows = c->n_rows;
    out->n_cols = c->n_cols;
    out->nnz = c->nnz;
    out->n_levels = -1;
    out->max_level_width = -1;
    // the longest chain is final when the build ends, which copied its info
    // words to the handle's pinned slot (complete once ev_use is): no device
    // read, so nothing here waits for other streams' copies
    out->max_chain = c->h_info[INFO_MAX_CHAIN];
    float ms = 0;
    if (c->timed_build && cudaEventElapsedTime(&ms, c->ev0, c->ev1) == cudaSuccess) out->ms_build = ms;
    if (c->timed_sgd && cudaEventElapsedTime(&ms, c->ev_sgd0, c->ev_sgd1) == cudaSuccess) out->ms_sgd = ms;
    if (c->timed_sgd && cudaEventElapsedTime(&ms, c->ev_k0, c->ev_k1) == cudaSuccess) out->ms_sgd_kernels = ms;
    if (c->timed_bsp && cudaEventElapsedTime(&ms, c->ev_bsp0, c->ev_bsp1) == cudaSuccess) out->ms_bsp = ms;
    out->sched_mode = -1;
    if (h) {
        out->sched_mode = h->mode;
        if (h->timed && cudaEventElapsedTime(&ms, h->ev0, h->ev1) == cudaSuccess) out->ms_schedule = ms;
        if (h->mode == PDB_SCHED_LEVELS) {
            LevelCtl ctl;
            if (read_words(&ctl, h->ctl, sizeof ctl) != PDB_OK) return PDB_ECUDA;
            out->n_levels = c->n_rows > 0 ? ctl.n_levels : 0;
            out->max_level_width = ctl.max_width;
        }
    }
    cudaGetLastError();
    return PDB_OK;
}

int pdb_memcpy(void *dst, const void *src, size_t bytes, void *stream)
{
    if (bytes == 0) return PDB_OK;
    if (!dst || !src) return PDB_EINVAL;
    return cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDefault, (cudaStream_t)stream) == cudaSuccess ? PDB_OK
                                                                                                 : PDB_ECUDA;
}

}  // extern "C"
