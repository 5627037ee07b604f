// Resident-weight chain engine: pdb_sgd_epoch under a CHAIN schedule whose
// examples are longer than the forwarding engine takes (256 ids) and whose
// n_cols weights all fit in one thread block's shared memory (about 55,000
// features with short rows, fewer with long ones).  For shorter rows the
// forwarding engine (chain.cu) was measured faster: random shared-memory
// reads and writes of w cost more than its forwarded slots.
//
// The conflict graph is close to one chain (or is one: with dense examples
// every example reads and writes every feature), so the examples run
// strictly in data order -- Algorithm 1 itself -- in one thread block, and
// w lives in shared memory for the whole call: an example reads w_j and
// writes w_j back with shared-memory accesses, in program order of the one
// computing warp.  No per-position link words, forwarding or write-through
// are needed, and rows may be as long as shared memory allows.
//
//   warp 0      computes example r: lane i mod 32 accumulates element i with
//               fused multiply-adds, the 32 partials combine in the
//               butterfly order (the same fp32 operations as every engine),
//               then w_j -= (eta*g) * x_j for its elements;
//   warps 1, 2  copy the ids and values of one example each, DS steps ahead,
//               in 16-byte cp.async pieces;
//   warp 3      copies row bounds L steps ahead.
//
// Epochs follow each other without a drain: the pipeline runs over the
// example sequence of all epochs.  No spin waits.
#include <cuda_runtime.h>

#include "common.cuh"

using namespace pdb;

namespace {

constexpr int RZ_THREADS = 128;
constexpr int RZ_G = 2;                 // examples per pipeline step
constexpr int RZ_NS = 8;                // example slots (power of two, >= (DS + 1) * G)
constexpr int RZ_DS = 3;                // steps between an example's copies and its compute
constexpr int RZ_L = RZ_DS + 3;         // steps between its row bounds' copy and its first use
constexpr int RZ_RP = 32;               // row-bound ring (power of two, > (L + 2) * G)
constexpr int RZ_U = 8;                 // elements per lane loaded ahead on long rows
static_assert(RZ_NS >= (RZ_DS + 1) * RZ_G && RZ_RP > (RZ_L + 2) * RZ_G, "rings too short");

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
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_wait_1() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }
__device__ __forceinline__ void st_shared(unsigned addr, float v)
{
    asm volatile("st.shared.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ void cp_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// elements [b - off, b + k) of a 4-byte array into dst: 16-byte pieces from
// the aligned position b - off when every source is 16-byte aligned (vec),
// the tail (or everything, without vec) one element at a time
__device__ __forceinline__ void cp_row(void *dst, const void *src, int64_t b, int k, int off, bool vec, int lane)
{
    const int64_t a0 = b - off;
    const int64_t a1 = vec ? ((b + k) & ~(int64_t)3) : a0;
    const int n16 = a1 > a0 ? (int)((a1 - a0) >> 2) : 0;
    for (int c = lane; c < n16; c += 32) cp16((uint32_t *)dst + 4 * c, (const uint32_t *)src + a0 + 4 * c);
    for (int64_t e = (a1 > b ? a1 : b) + lane; e < b + k; e += 32)
        cp4((uint32_t *)dst + (e - a0), (const uint32_t *)src + e);
}

// the butterfly combine of warp_combine (partial l plus partial l + half,
// for half = 16, 8, 4, 2, 1), evaluated from shared memory by every lane
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
    __syncwarp();   // every lane has read the partials before the next example writes them
    return v[0];
}

// shared-memory layout (bytes), all pieces 16-byte aligned
struct Layout {
    int64_t w, col, val, y, rp, part, total;
    int kcap;
};
__host__ __device__ __forceinline__ Layout layout(int64_t n_cols, int kcap)
{
    Layout L;
    L.kcap = kcap;
    L.w = 0;
    L.col = L.w + ((n_cols * 4 + 15) & ~(int64_t)15);
    L.val = L.col + (int64_t)RZ_NS * kcap * 4;
    L.y = L.val + (int64_t)RZ_NS * kcap * 4;
    L.rp = L.y + RZ_NS * 4 + 16;
    L.part = L.rp + RZ_RP * 16;
    L.total = L.part + 64 * 4;      // 32 partial sums, then 32 scratch words
    return L;
}

template <int R>
__global__ __launch_bounds__(RZ_THREADS, 1) void k_sgd_resident(int32_t n_rows, int64_t n_cols, int kcap,
                                                                const int64_t *__restrict__ row_ptr,
                                                                const int32_t *__restrict__ col,
                                                                const float *__restrict__ val,
                                                                const float *__restrict__ y, float *w, int loss,
                                                                float eta, int epochs, bool vec, int *status,
                                                                uint64_t *trace)
{
    extern __shared__ __align__(16) unsigned char smem_raw[];
    if (read_status(status)) return;
    const Layout Lo = layout(n_cols, kcap);
    float *ws = reinterpret_cast<float *>(smem_raw + Lo.w);
    int32_t *cs = reinterpret_cast<int32_t *>(smem_raw + Lo.col);
    float *vs = reinterpret_cast<float *>(smem_raw + Lo.val);
    float *ys = reinterpret_cast<float *>(smem_raw + Lo.y);
    int64_t *rp = reinterpret_cast<int64_t *>(smem_raw + Lo.rp);    // [RZ_RP][2]: bounds of an example
    float *part = reinterpret_cast<float *>(smem_raw + Lo.part);
    const unsigned dump = (unsigned)__cvta_generic_to_shared(part + 32 + (threadIdx.x & 31));
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    for (int64_t f = tid; f < n_cols; f += RZ_THREADS) ws[f] = w[f];
    __syncthreads();

    const int64_t total = (int64_t)epochs * n_rows;          // examples of all epochs, in order
    const int64_t steps = (total + RZ_G - 1) / RZ_G;
    for (int64_t t = -RZ_L; t <= steps; ++t) {
        if (warp == 3) {
            // row bounds of the examples of step t + L
            const int64_t rg = (t + RZ_L) * RZ_G + lane;
            if (lane < RZ_G && rg >= 0 && rg < total) {
                const int64_t r = rg % n_rows;
                cp8(&rp[2 * (rg & (RZ_RP - 1))], row_ptr + r);
                cp8(&rp[2 * (rg & (RZ_RP - 1)) + 1], row_ptr + r + 1);
            }
        } else if (warp >= 1) {
            // ids, values and label of example g = warp - 1 of step t + DS
            const int64_t rg = (t + RZ_DS) * RZ_G + (warp - 1);
            if (rg >= 0 && rg < total) {
                const int64_t b = rp[2 * (rg & (RZ_RP - 1))];
                const int k = (int)(rp[2 * (rg & (RZ_RP - 1)) + 1] - b);
                const int off = vec ? (int)(b & 3) : 0;
                const int slot = (int)(rg & (RZ_NS - 1));
                cp_row(cs + (int64_t)slot * kcap, col, b, k, off, vec, lane);
                if (val) cp_row(vs + (int64_t)slot * kcap, val, b, k, off, vec, lane);
                if (lane == 0) cp4(&ys[slot], y + rg % n_rows);
            }
        }
        if (warp != 0) {
            cp_commit();
            cp_wait_1();
        } else if (t >= 0 && t < steps) {
            for (int64_t rg = t * RZ_G; rg < min64(total, (t + 1) * RZ_G); ++rg) {
                const int64_t b = rp[2 * (rg & (RZ_RP - 1))];
                const int k = (int)(rp[2 * (rg & (RZ_RP - 1)) + 1] - b);
                const int off = vec ? (int)(b & 3) : 0;
                const int slot = (int)(rg & (RZ_NS - 1));
                const int32_t *ci = cs + (int64_t)slot * kcap + off;
                const float *vi = vs + (int64_t)slot * kcap + off;
                const float yr = ys[slot];
                float acc = 0.0f;
                if (k <= 32 * R) {
                    // the whole example in registers; no branches: lanes past the
                    // example's end read w_0 and store into a scratch word
                    int j[R];
                    float x[R], wv[R];
#pragma unroll
                    for (int q = 0; q < R; ++q) {
                        const int i = q * 32 + lane;
                        j[q] = i < k ? ci[i] : 0;
                        x[q] = i < k ? (val ? vi[i] : 1.0f) : 0.0f;
                    }
#pragma unroll
                    for (int q = 0; q < R; ++q) wv[q] = ws[j[q]];
#pragma unroll
                    for (int q = 0; q < R; ++q) {
                        const float f = __fmaf_rn(wv[q], x[q], acc);
                        acc = q * 32 + lane < k ? f : acc;
                    }
                    const float m = combine_smem(acc, part);
                    trace_mark(trace, rg, 0);
                    const float c = __fmul_rn(eta, dev_grad(loss, m, yr));
                    trace_mark(trace, rg, 1);   // before any write is visible
                    const unsigned ws_base = (unsigned)__cvta_generic_to_shared(ws);
#pragma unroll
                    for (int q = 0; q < R; ++q)
                        st_shared(q * 32 + lane < k ? ws_base + 4u * (unsigned)j[q] : dump,
                                  __fsub_rn(wv[q], __fmul_rn(c, x[q])));
                } else {
                    // long example, in pieces of RZ_U elements per lane (all their loads
                    // issued before the lane's fused multiply-adds, which keep element
                    // order); a second pass re-reads w_j (ids in a row are distinct, so
                    // no element of this example has changed another's weight)
                    for (int base = 0; base < k; base += 32 * RZ_U) {
                        float x[RZ_U], wv[RZ_U];
#pragma unroll
                        for (int u = 0; u < RZ_U; ++u) {
                            const int i = base + u * 32 + lane;
                            x[u] = 0.0f;
                            wv[u] = 0.0f;
                            if (i < k) {
                                x[u] = val ? vi[i] : 1.0f;
                                wv[u] = ws[ci[i]];
                            }
                        }
#pragma unroll
                        for (int u = 0; u < RZ_U; ++u)
                            if (base + u * 32 + lane < k) acc = __fmaf_rn(wv[u], x[u], acc);
                    }
                    const float m = combine_smem(acc, part);
                    trace_mark(trace, rg, 0);
                    const float c = __fmul_rn(eta, dev_grad(loss, m, yr));
                    trace_mark(trace, rg, 1);   // before any write is visible
                    for (int base = 0; base < k; base += 32 * RZ_U) {
                        int j[RZ_U];
                        float x[RZ_U], wv[RZ_U];
#pragma unroll
                        for (int u = 0; u < RZ_U; ++u) {
                            const int i = base + u * 32 + lane;
                            if (i < k) {
                                j[u] = ci[i];
                                x[u] = val ? vi[i] : 1.0f;
                                wv[u] = ws[j[u]];
                            }
                        }
#pragma unroll
                        for (int u = 0; u < RZ_U; ++u)
                            if (base + u * 32 + lane < k) ws[j[u]] = __fsub_rn(wv[u], __fmul_rn(c, x[u]));
                    }
                }
                __syncwarp();   // the next example may read these weights from another lane
            }
        }
        __syncthreads();
    }
    cp_wait_all();
    __syncthreads();
    for (int64_t f = tid; f < n_cols; f += RZ_THREADS) w[f] = ws[f];
}

int kcap_for(int64_t max_row) { return (int)(((max_row + 3) & ~(int64_t)3) + 4); }

}  // namespace

namespace pdb {

// shared memory this engine needs for n_cols weights and rows of max_row
// ids; 0 when it does not fit in one block
int64_t resident_smem(int64_t n_cols, int64_t max_row)
{
    if (n_cols < 1 || max_row < 0 || max_row > (1 << 20)) return 0;
    int dev = 0, optin = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    const int64_t bytes = layout(n_cols, kcap_for(max_row)).total;
    return bytes <= optin ? bytes : 0;
}

int resident_run(const pdb_csr *X, const float *y, float *w, int loss, float eta, int epochs, int max_row,
                 int *status, uint64_t *trace, cudaStream_t s)
{
    const int64_t smem = resident_smem(X->n_cols, max_row);
    if (smem == 0) return PDB_ETOOBIG;
    // registers per lane for the longest example: 1 .. 32 (32 to 1024 ids); longer rows
    // take the two-pass path of the 32-register variant
    auto kern = max_row <= 32 ? k_sgd_resident<1> : max_row <= 64 ? k_sgd_resident<2>
              : max_row <= 128 ? k_sgd_resident<4> : max_row <= 256 ? k_sgd_resident<8>
              : max_row <= 512 ? k_sgd_resident<16> : k_sgd_resident<32>;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
        return PDB_ECUDA;
    const bool vec = ((uintptr_t)X->col & 15) == 0 && ((uintptr_t)X->val & 15) == 0;
    kern<<<1, RZ_THREADS, (size_t)smem, s>>>((int32_t)X->n_rows, X->n_cols, kcap_for(max_row), X->row_ptr, X->col,
                                             X->val, y, w, loss, eta, epochs, vec, status, trace);
    note_launch();
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

}  // namespace pdb
