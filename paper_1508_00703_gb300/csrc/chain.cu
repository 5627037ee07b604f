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
//                values, labels and link words 5 steps ahead; the weights
//                nobody will push 3 steps ahead, together with the shared
//                memory address each new weight goes to), lanes striding
//                over the example's elements;
//   warps 6, 7   write the new weights of the previous step that are not
//                pushed through to global memory, and copy row bounds 9
//                steps ahead;
//   warp 4       only joins the barriers: warps map to the SM's four
//                schedulers by index mod 4, and warp 0 keeps its own.
//
// A pipeline step handles G = 4 consecutive examples, so the fixed cost of a
// step (barrier, copy bookkeeping) is shared by four hops.
//
// Ordering: a pushed weight (next occurrence within D = 20 examples) is
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

// Pipeline shape for rows of up to 32 R ids.  G examples per step, each
// prefetched by a warp of its own (a warp spends ~1500 cycles of issue on one
// example's copies per step, so rows of up to 128 ids take 8 per step);
// DS / BS = steps between the ids / weights prefetch and the compute; D = G *
// DS the forwarding window (examples); SLOTS example slots, RP row_ptr ring
// entries.  Rows of up to 256 ids take 4 per step, so their slots fit in
// shared memory.
template <int R>
struct ChainCfg {
    static constexpr int G = R <= 4 ? 8 : 4;
    static constexpr int DS = 5;
    static constexpr int BS = 3;
    static constexpr int INFLIGHT = 1;              // copy groups a prefetch warp leaves in flight at a step's end
    static constexpr int L = DS + BS + 1;           // steps between a row_ptr copy and its first use
    static constexpr int D = G * DS;
    static constexpr int SLOTS = R <= 4 ? 64 : 32;
    static constexpr int MAXK = 32 * R;             // longest example
    static constexpr int RP = 128;
    static constexpr int ROW = MAXK + 4;            // ids and link words of an example, from the aligned element before
    static constexpr int THREADS = R == 1 ? 768 : 512;
};
constexpr int CH_MAXK = 256;                        // longest example this engine takes
// link word of a position: bit 31 = its weight will be pushed by an earlier
// example (skip the gather); bit 30 = push the new weight to the next
// occurrence, which is element (bits 0..7) of the example (bits 16..23)
// examples later; bit 29 = the previous occurrence is in the example just
// before, as its element (bits 8..15)
constexpr uint32_t LK_RECV = 1u << 31, LK_PUSH = 1u << 30, LK_LATE = 1u << 29;
// store address word the compute warp reads per element: the shared-memory
// address of the new weight (below 2^22), bit 22 = the weight arrives from
// the example just before, as its element (bits 23..30)
constexpr uint32_t PA_ADDR = (1u << 22) - 1, PA_LATE = 1u << 22;
template <int R>
constexpr bool chain_cfg_ok()
{
    using C = ChainCfg<R>;
    return (C::SLOTS & (C::SLOTS - 1)) == 0 && (C::RP & (C::RP - 1)) == 0 &&   // rings are powers of two
           C::SLOTS > (C::DS + 2) * C::G && C::RP > (C::L + 2) * C::G + 1 &&  // and long enough
           C::D < 256 && C::MAXK <= 256 &&                                      // link word fields
           (C::G & (C::G - 1)) == 0 &&
           // a weight is gathered (not pushed) when its last writer r' lies more
           // than D examples back; r' stores it through at step r'/G + 1, the gather
           // for r runs at step r/G - BS, and r/G - r'/G >= (D + 1) / G: the store
           // lands at least one step (one __syncthreads) before the gather
           (C::D + 1) / C::G >= C::BS + 2 &&
           // the copies issued at step s complete by the end of step s + INFLIGHT,
           // so during step t the slots of steps up to t + BS - INFLIGHT - 1 are
           // complete: the compute warp for rows of up to 32 ids fetches the
           // first example of step t + 1 during step t
           C::BS - C::INFLIGHT - 1 >= 1 &&
           C::G <= 8;
}

static_assert(ChainCfg<8>::MAXK == CH_MAXK, "longest example");

// ids and link words are copied in 16-byte pieces from the aligned element
// before the example's first one: element i sits at index off + i, off =
// (first position) mod 4 (0 when an input array is not 16-byte aligned).
// Everything the compute warp reads is at element index i, so its loads need
// no row bounds.
template <int R>
struct ChainSmem {
    using C = ChainCfg<R>;
    int32_t col[C::SLOTS][C::ROW];
    uint32_t link[C::SLOTS][C::ROW];
    float xa[C::SLOTS][C::MAXK];    // value of each element (1 without values)
    uint32_t pa[C::SLOTS][C::MAXK]; // where the compute warp stores each element's new weight
    float wp[C::SLOTS][C::MAXK];    // weight each element reads (gathered or pushed)
    float out[C::SLOTS][C::MAXK];   // weight of the elements whose next occurrence is not pushed
    int64_t rp[C::RP];
    float y[C::SLOTS];
    int kk[C::SLOTS];               // length of each example
    float dump[2][32];              // store target of the lanes past an example's end
    __align__(16) float part[32];   // the compute warp's 32 partial sums
    float cbuf[2];                  // rows of up to 32 ids: c of each compute warp's last example,
    float wr[2][32], xr[2][32];     // and the weight read and value at each of its lanes
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
// Roles of the warps (scheduler = warp index mod 4).  Rows of up to 32 ids
// (24 warps): warps 0 and 1 compute, each alone on its scheduler (the other
// warps there only join the barriers, so nothing else issues or fetches
// instructions beside them); on schedulers 2 and 3, warps 2-15 prefetch one
// example g of a step each (ids, values, link words, then weights and store
// addresses) and warps 18, 19, 22, 23 write the weights of the previous step
// through (two examples each: gW = 0, 2, 4, 6; the first also copies row
// bounds).  Longer rows (16 warps): warp 0 computes alone on scheduler 0,
// and the warps of schedulers 1-3 in index order take the G prefetch roles
// and then the G / 2 write-through roles.  Returns g (prefetch = true) or gW
// (prefetch = false), -1 for none.
template <int R>
__host__ __device__ constexpr int chain_role(int warp, bool prefetch)
{
    using C = ChainCfg<R>;
    const int q = warp & 3, v = warp >> 2;
    if (R == 1) {
        const int k = q >= 2 ? (q - 2) * 6 + v : -1;       // 0..11 over the warps of schedulers 2, 3
        const int g = k >= 0 && k < 4 ? k : k >= 6 && k < 10 ? k - 2 : -1;
        const int wv = k == 4 ? 0 : k == 5 ? 2 : k == 10 ? 4 : k == 11 ? 6 : -1;
        if (prefetch) return g >= 0 && g < C::G ? g : -1;
        return wv >= 0 && wv < C::G ? wv : -1;
    }
    const int role = q ? warp - 1 - v : -1;
    if (prefetch) return role >= 0 && role < C::G ? role : -1;
    return role >= C::G && role < C::G + C::G / 2 ? 2 * (role - C::G) : -1;
}

// every prefetch role g < G and write-through role (even gW < G) taken by
// exactly one warp, none of them a compute warp
template <int R>
constexpr bool chain_roles_ok()
{
    using C = ChainCfg<R>;
    int seenA = 0, seenW = 0;
    for (int warp = 0; warp < C::THREADS / 32; ++warp) {
        const int a = chain_role<R>(warp, true), w = chain_role<R>(warp, false);
        if ((a >= 0 || w >= 0) && (warp == 0 || (R == 1 && warp == 1))) return false;
        if (a >= 0 && w >= 0) return false;
        if (a >= 0) {
            if (a >= C::G || (seenA >> a) & 1) return false;
            seenA |= 1 << a;
        }
        if (w >= 0) {
            if (w >= C::G || (w & 1) || (seenW >> w) & 1) return false;
            seenW |= 1 << w;
        }
    }
    return seenA == (1 << C::G) - 1 && seenW == 0x55 % (1 << C::G);
}
static_assert(chain_cfg_ok<1>() && chain_cfg_ok<2>() && chain_cfg_ok<4>() && chain_cfg_ok<8>(), "chain pipeline shape");
static_assert(chain_roles_ok<1>() && chain_roles_ok<2>() && chain_roles_ok<4>() && chain_roles_ok<8>(), "warp roles");

// named barriers between the two compute warps for rows of up to 32 ids
// (barrier 0 is __syncthreads): arrive marks this warp's arrival without
// waiting and orders its earlier shared-memory writes before the barrier
// completes; sync waits for the other warp's arrival
constexpr int BAR_C = 1, BAR_S = 3;     // + warp P: c published / stores done by P
__device__ __forceinline__ void bar_arrive2(int id) { asm volatile("bar.arrive %0, 64;" ::"r"(id) : "memory"); }
__device__ __forceinline__ void bar_sync2(int id) { asm volatile("bar.sync %0, 64;" ::"r"(id) : "memory"); }
__device__ __forceinline__ void st_shared(unsigned addr, float v)
{
    asm volatile("st.shared.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait_b() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }
__device__ __forceinline__ void cp_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// bounds [b, b + k) of example r from the row_ptr ring (false outside
// 0..N-1) and the offset of its elements in the 16-byte-copied rows
template <int R>
__device__ __forceinline__ bool row_bounds(const ChainSmem<R> &S, int r, int N, bool vec, int64_t &b, int &k, int &off)
{
    constexpr int RP = ChainCfg<R>::RP;
    if (r < 0 || r >= N) return false;
    b = S.rp[r & (RP - 1)];
    k = (int)(S.rp[(r + 1) & (RP - 1)] - b);
    off = vec ? (int)(b & 3) : 0;
    return true;
}

// ---- the compute warps for rows of at most 32 ids (one element per lane) ----
//
// Here the margin's 32 partial sums are single products, so an example's
// margin depends on the example just before only through its late elements
// (previous occurrence in that example), whose weights are w - c * x with
// that example's c.  Two warps take the examples in turn (warp 0 the even
// ones, warp 1 the odd ones, each on a scheduler of its own).
// While one computes example r's gradient, the other prepares r + 1: it
// fetches r + 1's slot, combines its other elements (late leaves as zero),
// and keeps for each lane the node its path adds at each level of the tree.
// When c of r arrives (through shared memory and a named barrier, with the
// weight and value r read at each lane), each lane forms its late weight
// itself (the same two roundings as the lane of r that stores it), and with
// at most two late elements every lane finishes the margin with five
// additions on the late paths -- the operands of the full tree, so the same
// bits.  With three or more, the whole tree is combined again.
//
// Hand-offs, per example r of warp P (the other warp is P' = P ^ 1):
//   bar CB_P  P arrives once c of r and the weights and values r read are in
//             shared memory; P' waits on it before example r + 1;
//   bar SB_P  P arrives once r's new weights are stored; P' waits on it
//             before it publishes c of r + 1 and fetches r + 3's slot.
// Each barrier has one arriving warp and one waiting warp (64 threads), and
// every arrival is matched by one wait: P arrives for r only when r + 1
// exists, and P' waits for r - 1 only when r > 0.  Arrivals and waits
// alternate: P's next arrival on either barrier needs c of r + 1, which P'
// publishes only after both of its waits for r.

// xor-butterfly combine in two exchange rounds: the first brings the leaves
// of lanes l ^ 16, 8, 24, 4, 20, 12, 28 and adds levels 1-3 locally, the
// second the level-3 nodes of lanes l ^ 2, 1, 3 and adds levels 4 and 5.
// Every addition has the operands that the one-level-per-shuffle butterfly
// gives it (node(l) + node(l ^ off); fp32 addition commutes), so the result
// has the same bits.  sib[t] is the node lane l's path adds at level t + 1
// (the other half of its level-(t + 1) subtree).
__device__ __forceinline__ float combine2(float a, float sib[5])
{
    const float b16 = __shfl_xor_sync(FULL, a, 16), b8 = __shfl_xor_sync(FULL, a, 8);
    const float b24 = __shfl_xor_sync(FULL, a, 24), b4 = __shfl_xor_sync(FULL, a, 4);
    const float b20 = __shfl_xor_sync(FULL, a, 20), b12 = __shfl_xor_sync(FULL, a, 12);
    const float b28 = __shfl_xor_sync(FULL, a, 28);
    const float n1 = __fadd_rn(a, b16);                                     // level 1
    const float n1x8 = __fadd_rn(b8, b24);                                  // level 1 of lane l ^ 8
    const float n2x4 = __fadd_rn(__fadd_rn(b4, b20), __fadd_rn(b12, b28));  // level 2 of lane l ^ 4
    const float n3 = __fadd_rn(__fadd_rn(n1, n1x8), n2x4);                  // levels 2, 3
    const float c2 = __shfl_xor_sync(FULL, n3, 2), c1 = __shfl_xor_sync(FULL, n3, 1);
    const float c3 = __shfl_xor_sync(FULL, n3, 3);
    const float n4x1 = __fadd_rn(c1, c3);                                   // level 4 of lane l ^ 1
    sib[0] = b16;
    sib[1] = n1x8;
    sib[2] = n2x4;
    sib[3] = c2;
    sib[4] = n4x1;
    return __fadd_rn(__fadd_rn(n3, c2), n4x1);                              // levels 4, 5
}

// one example in the R = 1 pipeline (registers of the compute warp)
struct Ex1 {
    float x, wv, y;         // this lane's value and slot weight; the label
    unsigned pa;            // store word
    int k;                  // length
    bool late;              // this lane's element is late
    int src;                // lane of its previous occurrence
    int K, d;               // late elements; level (1-5) at which two late paths meet
    float me;               // margin when no element is late
    float sA[5], sB[4];     // node the first / second late element's path adds per level
    float x1, x2;           // values of the first two late elements, in every lane
    int src1, src2;         // lanes of their previous occurrences
};

template <int R>
__device__ __forceinline__ void fetch1(const ChainSmem<R> &S, int r, int lane, Ex1 &e)
{
    const int slot = r & (ChainCfg<R>::SLOTS - 1);
    e.k = S.kk[slot];
    e.y = S.y[slot];
    e.x = S.xa[slot][lane];
    e.pa = S.pa[slot][lane];
    e.wv = S.wp[slot][lane];
}

// everything of example e that does not wait for the example before it
__device__ __forceinline__ void early1(Ex1 &e, int lane)
{
    const bool act = lane < e.k;
    e.late = act && (e.pa & PA_LATE);
    const unsigned bal = __ballot_sync(FULL, e.late);
    e.K = __popc(bal);
    const int k1 = (__ffs(bal) - 1) & 31;              // lanes of the first two late elements
    const int k2 = (__ffs(bal & (bal - 1)) - 1) & 31;
    // two leaves share their level-t subtree once the xor of their lanes has
    // no set bit below 5 - t
    e.d = e.K == 2 ? 6 - __ffs(k1 ^ k2) : 0;
    e.src = (int)((e.pa >> 23) & 31u);
    e.src1 = __shfl_sync(FULL, e.src, k1);
    e.src2 = __shfl_sync(FULL, e.src, k2);
    e.x1 = __shfl_sync(FULL, e.x, k1);
    e.x2 = __shfl_sync(FULL, e.x, k2);
    float sib[5];
    e.me = combine2(act && !e.late ? __fmaf_rn(e.wv, e.x, 0.0f) : 0.0f, sib);
#pragma unroll
    for (int t = 0; t < 5; ++t) e.sA[t] = __shfl_sync(FULL, sib[t], k1);
#pragma unroll
    for (int t = 0; t < 4; ++t) e.sB[t] = __shfl_sync(FULL, sib[t], k2);
}

// margin of e once c of the example before it is known: wc = this lane's
// weight; (wo1, xo1), (wo2, xo2) = weight read and value of the first two late
// elements' previous occurrences
__device__ __forceinline__ float margin1(const Ex1 &e, float c, float wc, int lane, float wo1, float xo1, float wo2,
                                         float xo2)
{
    if (e.K <= 2) {
        float A = __fmaf_rn(__fsub_rn(wo1, __fmul_rn(c, xo1)), e.x1, 0.0f);
        float B = __fmaf_rn(__fsub_rn(wo2, __fmul_rn(c, xo2)), e.x2, 0.0f);
#pragma unroll
        for (int t = 0; t < 5; ++t) {
            A = __fadd_rn(A, e.d == t + 1 ? B : e.sA[t]);
            if (t < 4) B = __fadd_rn(B, e.sB[t]);
        }
        return e.K == 0 ? e.me : A;
    }
    float sib[5];
    return combine2(lane < e.k ? __fmaf_rn(wc, e.x, 0.0f) : 0.0f, sib);
}

template <int R, int LOSS, bool TRACE>
__global__ __launch_bounds__(ChainCfg<R>::THREADS, 1) void k_sgd_chain(int32_t n_rows, const int64_t *__restrict__ row_ptr,
                                                             const int32_t *__restrict__ col,
                                                             const float *__restrict__ val,
                                                             const float *__restrict__ y,
                                                             const uint32_t *__restrict__ link, float *w, int loss,
                                                             float eta, int epochs, bool vec, int *status,
                                                             uint64_t *trace)
{
    using C = ChainCfg<R>;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    ChainSmem<R> &S = *reinterpret_cast<ChainSmem<R> *>(smem_raw);
    if (read_status(status)) return;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // Warps map to the SM's four schedulers by index mod 4; each warp's role
    // is chain_role's.
    const bool compute = warp == 0 || (R == 1 && warp == 1);
    const int P = warp & 1;         // compute warp 0 or 1 (rows of up to 32 ids)
    const unsigned wp_base = (unsigned)__cvta_generic_to_shared(&S.wp[0][0]);
    const unsigned out_base = (unsigned)__cvta_generic_to_shared(&S.out[0][0]);
    const int gA = chain_role<R>(warp, true), gW = chain_role<R>(warp, false);
    const int N = n_rows;
    const int steps = (N + C::G - 1) / C::G;
    // R = 1 compute state carried from example to example (warp 0 only): the
    // next example, c of the one before and its weights, values and store
    // addresses, whose stores wait for the next example's margin to start
    Ex1 E;      // rows of up to 32 ids: this compute warp's next example

    for (int ep = 0; ep < epochs; ++ep) {
        for (int t = -C::L; t <= steps; ++t) {
            if (gW >= 0) {
                // stage W: new weights of step t - 1 that no example among the next D takes
                // on chip go through to global memory (a pushed weight is re-written by its
                // receiver, so two stores of one step never hit one address)
                for (int g = gW; g < gW + 2; ++g) {
                    const int r = (t - 1) * C::G + g;
                    int64_t b;
                    int k, off;
                    if (row_bounds(S, r, N, vec, b, k, off)) {
                        const int slot = r & (C::SLOTS - 1);
                        for (int i = lane; i < k; i += 32)
                            if (!(S.link[slot][off + i] & LK_PUSH)) w[S.col[slot][off + i]] = S.out[slot][i];
                    }
                }
                // stage R: row_ptr entries [(t+L)G, (t+L)G + G) with L = DS + BS + 1, so that
                // stage A of step t finds the bounds of step t + DS (and the entry after it) complete
                if (gW == 0 && lane < C::G) {
                    const int r = (t + C::L) * C::G + lane;
                    if (r >= 0 && r <= N) cp8(&S.rp[r & (C::RP - 1)], row_ptr + r);
                }
            } else if (gA >= 0) {
                // stage A: ids, values, link words and label of example g of step t + DS
                {
                    const int r = (t + C::DS) * C::G + gA;
                    int64_t b;
                    int k, off;
                    if (row_bounds(S, r, N, vec, b, k, off)) {
                        const int slot = r & (C::SLOTS - 1);
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
                    const int r = (t + C::BS) * C::G + gA;
                    int64_t b;
                    int k, off;
                    if (row_bounds(S, r, N, vec, b, k, off)) {
                        const int slot = r & (C::SLOTS - 1);
                        for (int i = lane; i < k; i += 32) {
                            const uint32_t lk = S.link[slot][off + i];
                            if (!(lk & LK_RECV)) cp4(&S.wp[slot][i], w + S.col[slot][off + i]);
                            const unsigned tslot = ((unsigned)r + ((lk >> 16) & 0xffu)) & (C::SLOTS - 1);
                            const unsigned addr = (lk & LK_PUSH) ? wp_base + 4u * (tslot * C::MAXK + (lk & 0xffu))
                                                                 : out_base + 4u * ((unsigned)slot * C::MAXK + i);
                            S.pa[slot][i] = addr | ((lk & LK_LATE) ? PA_LATE | (((lk >> 8) & 0xffu) << 23) : 0u);
                        }
                        if (lane == 0) S.kk[slot] = k;
                    }
                }
            }
            if (!compute) {
                cp_commit();
                cp_wait_b<C::INFLIGHT>();
            } else if (t >= 0 && t < steps) {
              if constexpr (R == 1) {
                // this warp's examples of step t (every other one), in data order
                const int r0 = t * C::G, r1 = min(N, r0 + C::G);
                const unsigned dump = (unsigned)__cvta_generic_to_shared(&S.dump[P][lane]);
                if (t == 0) {
                    // the first example of the epoch (0 has no example before it)
                    fetch1(S, P, lane, E);
                    early1(E, lane);
                }
                for (int r = r0 + P; r < r1; r += 2) {
                    // c of r - 1 and the weight and value it read at each lane
                    if (r > 0) bar_sync2(BAR_C + (P ^ 1));
                    const float c_prev = S.cbuf[P ^ 1];
                    const float wo = S.wr[P ^ 1][E.src], xo = S.xr[P ^ 1][E.src];
                    const float wo1 = S.wr[P ^ 1][E.src1], xo1 = S.xr[P ^ 1][E.src1];
                    const float wo2 = S.wr[P ^ 1][E.src2], xo2 = S.xr[P ^ 1][E.src2];
                    // this lane's weight: a late one from r - 1's c; r + 1 takes it from here
                    const float wc = E.late ? __fsub_rn(wo, __fmul_rn(c_prev, xo)) : E.wv;
                    S.wr[P][lane] = wc;
                    S.xr[P][lane] = E.x;
                    if (TRACE) trace_mark(trace, (int64_t)ep * N + r, 0);    // every weight is read
                    const float m = margin1(E, c_prev, wc, lane, wo1, xo1, wo2, xo2);
                    const float c = dev_step(LOSS, m, E.y, eta);
                    if (TRACE) trace_mark(trace, (int64_t)ep * N + r, 1);    // before any write is visible
                    // r - 1's stores are done before r + 1 may start (and before this
                    // warp fetches r + 2, whose slot they complete)
                    if (r > 0) bar_sync2(BAR_S + (P ^ 1));
                    if (r + 1 < N) {
                        S.cbuf[P] = c;
                        bar_arrive2(BAR_C + P);
                    }
                    // r's new weights: pushed into a later example's slot, or kept for
                    // write-through by the W warps in the next step
                    st_shared(lane < E.k ? (E.pa & PA_ADDR) : dump, __fsub_rn(wc, __fmul_rn(c, E.x)));
                    if (r + 1 < N) bar_arrive2(BAR_S + P);
                    __syncwarp();
                    // this warp's next example, r + 2
                    fetch1(S, r + 2, lane, E);
                    early1(E, lane);
                }
              } else {
                // compute the G examples of step t in data order.  The first takes every
                // weight from its slot.  Each later one fetches its length, label, values,
                // store words and weights while the example before computes its gradient:
                // a weight that example writes (its previous occurrence is there) is taken
                // from it once it exists -- by shuffle from the lane that computed it for
                // rows of up to 64 ids, else from the slot after the pushes are stored --
                // and every other weight is final when fetched.
                const int r0 = t * C::G, r1 = min(N, r0 + C::G);
                const unsigned dump = (unsigned)__cvta_generic_to_shared(&S.dump[0][lane]);
                int k;
                float yr, xv[R], wv[R];
                unsigned pa[R];
                auto fetch = [&](int r) {
                    const int slot = r & (C::SLOTS - 1);
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
                        const int nslot = (r + 1) & (C::SLOTS - 1);
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
            }
            __syncthreads();
        }
        cp_wait_all();
        __syncthreads();
    }
}

// link[p] (layout above): receive flag from the previous occurrence, push
// target from the next occurrence, each when it lies within D examples
__global__ void k_chain_link(const int32_t *__restrict__ prev, const int32_t *__restrict__ next,
                             const int32_t *__restrict__ row_of, const int64_t *__restrict__ row_ptr, int64_t nnz,
                             uint32_t *__restrict__ link, int D, const int *status)
{
    if (read_status(status)) return;
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < nnz; p += (int64_t)gridDim.x * blockDim.x) {
        const int32_t t = row_of[p], q = prev[p], n = next[p];
        uint32_t l = 0;
        if (q >= 0 && t - row_of[q] <= D) l |= LK_RECV;
        if (q >= 0 && row_of[q] == t - 1) l |= LK_LATE | ((uint32_t)(q - row_ptr[t - 1]) << 8);
        if (n >= 0) {
            const int32_t tn = row_of[n];
            if (tn - t <= D) l |= LK_PUSH | ((uint32_t)(tn - t) << 16) | (uint32_t)(n - row_ptr[tn]);
        }
        link[p] = l;
    }
}

}  // namespace

namespace pdb {

int chain_max_row() { return CH_MAXK; }

// registers per lane for the longest example: 1, 2, 4 or 8 (32 to 256 ids)
static int chain_regs(int64_t max_row) { return max_row <= 32 ? 1 : max_row <= 64 ? 2 : max_row <= 128 ? 4 : 8; }

int chain_schedule(const int32_t *prev, const int32_t *next, const int32_t *row_of, const int64_t *row_ptr,
                   int64_t nnz, int64_t max_row, uint32_t *link, const int *status, cudaStream_t s)
{
    // the forwarding window of the kernel that will run these rows
    const int R = chain_regs(max_row);
    const int D = R == 1 ? ChainCfg<1>::D : R == 2 ? ChainCfg<2>::D : R == 4 ? ChainCfg<4>::D : ChainCfg<8>::D;
    if (nnz > 0) {
        k_chain_link<<<grid_1d(nnz), 256, 0, s>>>(prev, next, row_of, row_ptr, nnz, link, D, status);
        note_launch();
    }
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

using ChainKernel = void (*)(int32_t, const int64_t *, const int32_t *, const float *, const float *,
                             const uint32_t *, float *, int, float, int, bool, int *, uint64_t *);

template <int R, bool TRACE>
static ChainKernel chain_kernel(int loss)
{
    return loss == PDB_LOSS_LOGISTIC ? k_sgd_chain<R, PDB_LOSS_LOGISTIC, TRACE>
           : loss == PDB_LOSS_SQUARED ? k_sgd_chain<R, PDB_LOSS_SQUARED, TRACE>
                                      : k_sgd_chain<R, PDB_LOSS_HINGE, TRACE>;
}

int chain_run(const pdb_csr *X, const float *y, const uint32_t *link, float *w, int loss, float eta, int epochs,
              int max_row, int *status, uint64_t *trace, cudaStream_t s)
{
    // one kernel per register count (chain_regs) and loss, so the gradient has
    // no branch; rows of up to 32 ids take the execution-trace stamps in a
    // kernel of their own (the others test the trace pointer at run time)
    const int R = chain_regs(max_row);
    const int rw = R == 1 ? (trace ? 4 : 0) : R == 2 ? 1 : R == 4 ? 2 : 3;
    const size_t smem = R == 1 ? sizeof(ChainSmem<1>) : R == 2 ? sizeof(ChainSmem<2>)
                        : R == 4 ? sizeof(ChainSmem<4>) : sizeof(ChainSmem<8>);
    const int threads = R == 1 ? ChainCfg<1>::THREADS : ChainCfg<2>::THREADS;
    const ChainKernel kern = rw == 0 ? chain_kernel<1, false>(loss) : rw == 4 ? chain_kernel<1, true>(loss)
                             : rw == 1 ? chain_kernel<2, false>(loss) : rw == 2 ? chain_kernel<4, false>(loss)
                                                                       : chain_kernel<8, false>(loss);
    const int variant = rw * 3 + (loss >= 0 && loss <= 2 ? loss : 2);
    // set once per device and variant (any device past the table: every call)
    static std::atomic<bool> configured[64][15];
    int dev = 0;
    cudaGetDevice(&dev);
    const bool known = dev >= 0 && dev < 64;
    if (!known || !configured[dev][variant].load(std::memory_order_acquire)) {
        if (cudaFuncSetAttribute((const void *)kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem) != cudaSuccess)
            return PDB_ECUDA;
        if (known) configured[dev][variant].store(true, std::memory_order_release);
    }
    // 16-byte row copies need 16-byte aligned ids, values and link words
    const bool vec = ((uintptr_t)X->col & 15) == 0 && ((uintptr_t)X->val & 15) == 0 && ((uintptr_t)link & 15) == 0;
    kern<<<1, threads, smem, s>>>((int32_t)X->n_rows, X->row_ptr, X->col, X->val, y, link, w, loss,
                                                  eta, epochs, vec, status, trace);
    note_launch();
    return cudaPeekAtLastError() == cudaSuccess ? PDB_OK : PDB_ECUDA;
}

}  // namespace pdb
