// vsd_lmhead_bwd.cu -- the draft LM head's backward on the tensor cores.  The
// gradient of the VSD objective (Algorithm 1's M-step) with respect to the
// draft logits x is kept in the factored form the fused E-step + M-step leaves
// in its workspace,
//
//   G[r][v] = gq_r 2^{(x_rv - m_r) c} - c0_r [v = t0_r] - c1_r [v = t1_r]
//             (+ the row's top-K terms of VSD (KL)),
//
// with m_r the row maximum, gq_r = g_r / Z_r the dense factor and c = log2(e)/T,
// and is carried into the head's two weight-side products:
//
//   d_hidden = G . W        [R][H]   (M = R, N = H, K = V)
//   d_weight = G^T . hidden [V][H]   (M = V, N = H, K = R)
//
// The A operand (G, or G^T) is made in shared memory from the TMA-loaded
// logits tile, element by element with the arithmetic of the E-step's
// gradient jobs (so each element rounds to the bf16 value those jobs write),
// right before the tensor cores read it: the dense gradient never goes to HBM.
// W and hidden are read as they lie, as MN-major B operands (no transposes),
// and so is the logits tile of d_weight as an MN-major A operand.
//
// One persistent CTA per SM computes 128 x (256 NT) output tiles (NT = 2: a
// tile fills the 512 TMEM columns), K in blocks of KB (32) through a ring of
// shared-memory stages:
//   warp 0          TMA producer: the logits tile and the B tile of each K
//                   block (for d_weight also the block's row factors);
//   warp 1          MMA issuer: one thread issues tcgen05.mma (kind::f16,
//                   M = 128, N = 256, K = 16; NT of them per K step, sharing
//                   A) into TMEM;
//   warps 2 .. 17   transform: the logits tile becomes the A operand in place;
//   the last 4      epilogue: tcgen05.ld of the accumulator, fp32 stores.
// d_hidden's 256 tiles at the lmhead sizes would leave a third of the SMs
// idle in a second wave, so there the (tile, K block) units are shared out
// evenly (stream-K) and tiles split between two CTAs are added into the
// zeroed output.  Every wait is bounded; a wait that runs out sets
// VSD_STATUS_TIMEOUT in the status word and the CTA winds down (waiting,
// again bounded, for its copies and MMAs in flight) and frees its tensor
// memory.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "vsd.h"
#include "vsd_launch.h"
#include "vsd_tc.cuh"

namespace vsd_bwd {

using namespace vsd_lm;
using vsd::Coef;
using vsd::KlRec;
using vsd::RowRec;

constexpr int BM = 128, BN = 256;
#ifndef VSD_BWD_XWARPS
#define VSD_BWD_XWARPS 16
#endif
// warps: 0 TMA, 1 MMA, 2 .. 2 + kXWarps - 1 transform, the last 4 epilogue
constexpr int kXWarps = VSD_BWD_XWARPS;
static_assert(kXWarps == 4 || kXWarps == 8 || kXWarps == 16, "a whole share of chunks per thread");
constexpr int kThreads = 32 * (kXWarps + 6);
#ifndef VSD_BWD_XGROUPS
#define VSD_BWD_XGROUPS 1
#endif
// The transform warps form up to kXGroups groups, so that several stages are
// made at once.  Stage s belongs to group s % groups: a group makes every
// round of its stages, in order, so that it never waits on a barrier phase
// more than one ahead of the barrier (a parity wait cannot tell those apart).
constexpr int kXGroups = VSD_BWD_XGROUPS;
static_assert(kXWarps % kXGroups == 0, "whole groups");
constexpr int kTmemCols = 512;
constexpr int kSmemMax = 232448;  // 227 KB of dynamic shared memory per block
constexpr int kMaxStages = 8;
enum Mode { kDHidden = 0, kDWeight = 1 };

// A row's gradient factors, packed from the E-step's records by k_rowfac.
struct __align__(16) Fac {
    float mx, gq, c0, c1;  // row maximum; g / Z; the two sparse terms
    int t0, t1, nkl;       // their tokens; top-K terms in the row's KL record
    int flags;             // kValid: a row of the problem; kDense: g q(v) is formed
};
static_assert(sizeof(Fac) == 32, "Fac layout");
constexpr int kValid = 1, kDense = 2;

// NT: 256-column MMAs per output tile (tile 128 x 256 NT); KB: K block (32 or
// 64 elements).  A stage holds the A tile (128 x KB, the logits tile made in
// place) and the B tile (256 NT x KB as 64-column boxes of KB rows).
// kDWeight stages also hold the K block's KB row factors (kFacBytes).
template <int MODE, int NT, int KB> struct Cfg {
    static_assert(KB == 32 || KB == 64, "K block");
    static constexpr int kABytes = BM * KB * 2;
    static constexpr int kBoxBytes = 64 * KB * 2;  // one 64-column box of KB rows
    static constexpr int kBBytes = NT * BN * KB * 2;
    static constexpr int kFacBytes = MODE == kDWeight ? KB * (int)sizeof(Fac) : 0;
    static constexpr int kStageBytes = kABytes + kBBytes + ((kFacBytes + 1023) & ~1023);
    static constexpr int kFit0 = (kSmemMax - 2048) / kStageBytes;
    static constexpr int kFit = kFit0 < kMaxStages ? kFit0 : kMaxStages;
    static constexpr int kGroups = kXGroups < kFit ? kXGroups : kFit;
    static constexpr int kGroupWarps = kXWarps / kGroups;
    static constexpr int kStages = kFit / kGroups * kGroups;  // whole rounds of the groups
    static constexpr int kAccBufs = NT == 1 ? 2 : 1;  // TMEM: 512 columns either way
    static_assert(kStages >= 2, "two stages at least");
};

struct Bars {
    uint64_t full[kMaxStages];   // TMA bytes landed
    uint64_t xform[kMaxStages];  // the A operand is made (one arrival per transform warp)
    uint64_t empty[kMaxStages];  // the MMAs reading the stage are done
    uint64_t acc_full[2];
    uint64_t acc_empty[2];  // 4 epilogue warp arrivals
    uint64_t drain;
    uint64_t timeout_ns;
    uint32_t tmem_base;
    int err;
};
static_assert(sizeof(Bars) <= 1024, "the barriers take the first 1 KB");
// [alignment pad][barriers: 1 KB][stages, 1024-byte aligned]
template <int MODE, int NT, int KB> constexpr size_t smem_bytes() {
    return 2048 + (size_t)Cfg<MODE, NT, KB>::kStages * Cfg<MODE, NT, KB>::kStageBytes;
}

__device__ __forceinline__ bool wait_phase(uint64_t* bar, uint32_t parity, Bars* sb, int* status) {
    return wait_phase_err(bar, parity, &sb->err, sb->timeout_ns, status);
}
// The same wait by a whole warp, with one outcome for all its lanes (a lane
// that gave up while another saw the phase complete would split the warp
// between the loop's __syncwarp and the final __syncthreads).
__device__ __forceinline__ bool wait_phase_warp(uint64_t* bar, uint32_t parity, Bars* sb,
                                                int* status) {
    return __all_sync(0xffffffffu, wait_phase(bar, parity, sb, status));
}

// Shared-memory descriptor of an MN-major bf16 operand in the 128-byte
// swizzle: 8-row K groups of 128-byte rows (64 MN elements) 1024 bytes apart
// (stride byte offset), 64-element MN blocks `lbo` bytes apart (leading byte
// offset), descriptor version 1, swizzle mode 2.
__device__ __forceinline__ uint64_t sdesc_mn_sw128(uint32_t saddr, uint32_t lbo) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)(1024 >> 4) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// Shared-memory descriptor of a K-major bf16 tile with 32-element (64-byte)
// rows in the 64-byte swizzle: 8-row groups 512 bytes apart (stride byte
// offset), the leading byte offset unused, version 1, swizzle mode 4.  A K
// step of 16 elements advances the start address by 32 bytes.
__device__ __forceinline__ uint64_t sdesc_sw64(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;
    d |= (uint64_t)(512 >> 4) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)4 << 61;
    return d;
}

// The persistent loop's work, segments (tile t, K blocks kb0 .. kb1 - 1).
// Tile mode: whole tiles blockIdx.x, blockIdx.x + gridDim.x, ...  Stream-K
// mode: the units (tile, K block) in tile order are shared out evenly, CTA c
// taking units [c U / G, (c + 1) U / G); a share is at least one tile long,
// so at most two CTAs meet on a tile and add into the zeroed output.
struct Seg {
    int t, kb0, kb1;
};
template <bool SK> struct SegIter {
    long long u, u1;  // stream-K: the next unit and the end of this CTA's share
    int t, nk, ntiles;
    __device__ SegIter(int ntiles_, int nk_) : nk(nk_), ntiles(ntiles_) {
        const long long U = (long long)ntiles_ * nk_;
        u = SK ? U * blockIdx.x / gridDim.x : 0;
        u1 = SK ? U * (blockIdx.x + 1) / gridDim.x : 0;
        t = blockIdx.x;
    }
    __device__ bool next(Seg& g) {
        if (!SK) {
            if (t >= ntiles) return false;
            g = Seg{t, 0, nk};
            t += gridDim.x;
            return true;
        }
        if (u >= u1) return false;
        g.t = (int)(u / nk);
        g.kb0 = (int)(u - (long long)g.t * nk);
        g.kb1 = (int)min((long long)nk, u1 - (long long)g.t * nk);
        u = (long long)g.t * nk + g.kb1;
        return true;
    }
};

#ifndef VSD_BWD_NFAST
#define VSD_BWD_NFAST 1
#endif
// Tile t of the persistent loop: with the N index fastest, the CTAs working at
// once share their A rows (read once from HBM, then from L2).
__device__ __forceinline__ void tile_origin(int t, int mt, int ntn, int tn, int& m0, int& n0) {
    const int mi = VSD_BWD_NFAST ? t / ntn : t % mt;
    const int ni = VSD_BWD_NFAST ? t % ntn : t / mt;
    m0 = mi * BM;
    n0 = ni * tn;
}

__global__ void k_rowfac(const RowRec* __restrict__ rows, const Coef* __restrict__ coef,
                         const KlRec* __restrict__ klr, int R, Fac* __restrict__ fac) {
    const int r = blockIdx.x * blockDim.x + threadIdx.x;
    if (r >= R) return;
    const float mx = rows[r].mx, izx = rows[r].izx;
    const Coef cf = coef[r];
    Fac f;
    f.mx = mx;
    f.gq = cf.g * izx;  // g / Z, as the gradient jobs form it
    f.c0 = cf.c0;
    f.c1 = cf.c1;
    f.t0 = cf.t0;
    f.t1 = cf.t1;
    f.nkl = klr ? min(max(klr[r].n, 0), vsd::kMaxKlTop) : 0;
    // no dense part where g = 0 and the row maximum is finite: g q(v) is +0
    f.flags = kValid | ((cf.g == 0.f && isfinite(mx)) ? 0 : kDense);
    fac[r] = f;
}

__device__ __forceinline__ Fac no_row() {
    Fac f;
    f.mx = f.gq = f.c0 = f.c1 = 0.f;
    f.t0 = f.t1 = -1;
    f.nkl = 0;
    f.flags = 0;
    return f;
}

// One gradient element, in the order of the E-step's gradient jobs: the dense
// part, minus the two sparse terms, plus the row's top-K terms.
__device__ __forceinline__ float grad_elem(float x, int v, const Fac& f, float c,
                                           const KlRec* kl) {
    // (rounded steps: no contraction into a fused multiply-add)
    float o = (f.flags & kDense) ? __fmul_rn(vsd::ex2(__fmul_rn(__fsub_rn(x, f.mx), c)), f.gq)
                                 : 0.f;
    if (v == f.t0) o = __fsub_rn(o, f.c0);
    if (v == f.t1) o = __fsub_rn(o, f.c1);
    for (int k = 0; k < f.nkl; ++k)
        if (v == __ldg(&kl->tok[k])) o = __fadd_rn(o, __ldg(&kl->coef[k]));
    return o;
}

// Bit j set: the 8 elements [vb + 8j, vb + 8j + 8) of the W elements from vb
// hold a sparse term or run past the vocabulary; they take the per-element
// path.
template <int W>
__device__ __forceinline__ uint32_t slow_chunks(const Fac& f, const KlRec* kl, int vb, int V) {
    uint32_t m = 0;
    auto mark = [&](int t) {
        const int d = t - vb;
        if ((unsigned)d < (unsigned)W) m |= 1u << (d >> 3);
    };
    mark(f.t0);
    mark(f.t1);
    for (int k = 0; k < f.nkl; ++k) mark(__ldg(&kl->tok[k]));
    if (vb + W > V) {
        const int first = V - vb;  // first chunk with an element past V
        for (int j = max(first, 0) >> 3; j < W / 8; ++j) m |= 1u << j;
    }
    return m;
}

// 8 logits (one 16-byte chunk of the tile, elements v0 .. v0 + 7 of row f)
// -> 8 bf16 gradient elements, in place.
__device__ __forceinline__ void make_chunk(uint4* cp, const Fac& f, float c, const KlRec* kl,
                                           int v0, int V, bool slow) {
    if (!(f.flags & kValid)) {
        *cp = make_uint4(0u, 0u, 0u, 0u);
        return;
    }
    const uint4 raw = *cp;
    const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
    uint32_t o[4];
    if (!slow) {
        const uint64_t mx2 = vsd::f2(f.mx, f.mx), c2 = vsd::f2(c, c), gq2 = vsd::f2(f.gq, f.gq);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            float lo = 0.f, hi = 0.f;
            if (f.flags & kDense)
                vsd::f2split(vsd::f2mul(vsd::f2_mass(vsd::bf16x2_pair(w[e]), mx2, c2), gq2), lo,
                             hi);
            const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
            o[e] = *reinterpret_cast<const uint32_t*>(&h);
        }
    } else {
        // (unrolled: constant indices keep w and o in registers)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int v = v0 + 2 * e;
            const float lo = v < V ? grad_elem(__uint_as_float(w[e] << 16), v, f, c, kl) : 0.f;
            const float hi =
                v + 1 < V ? grad_elem(__uint_as_float(w[e] & 0xFFFF0000u), v + 1, f, c, kl) : 0.f;
            const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
            o[e] = *reinterpret_cast<const uint32_t*>(&h);
        }
    }
    *cp = make_uint4(o[0], o[1], o[2], o[3]);
}

// ------------------------------------------------------------ the GEMMs
// MODE kDHidden: out[R][H] = G . W.  The A tile is x[m0 .. m0+127][k0 .. k0+KB)
// (K-major, one box; 128-byte swizzle for KB = 64, 64-byte for KB = 32); B is
// W[k0 .. k0+KB)[n0 .. n0 + 256 NT) read MN-major, 64-column boxes.
// MODE kDWeight: out[V][H] = G^T . hidden.  The A tile is x[k0 .. k0+KB)[m0 ..
// m0+127] read MN-major (two 64-column boxes); B is hidden[k0 .. k0+KB)[n0 ..)
// read MN-major like W above.
template <int MODE, int NT, int KB, bool SK>
__global__ void __launch_bounds__(kThreads, 1)
    k_lmhead_bwd(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmB,
                 const Fac* __restrict__ fac, const KlRec* __restrict__ klr, float c, int R,
                 int V, int H, float* __restrict__ out, int* status, uint64_t timeout_ns) {
    using C = Cfg<MODE, NT, KB>;
    constexpr int S = C::kStages;
    constexpr int TN = BN * NT;
    constexpr int kBox = C::kBoxBytes;
    // A MN-major in kDWeight (bit 15), B MN-major always (bit 16)
    constexpr uint32_t kIdesc =
        idesc_bf16(BM, BN) | (MODE == kDWeight ? (1u << 15) : 0u) | (1u << 16);
    extern __shared__ unsigned char dsm_raw[];
    unsigned char* base = dsm_raw + ((1024u - (smem_u32(dsm_raw) & 1023u)) & 1023u);
    Bars* sb = reinterpret_cast<Bars*>(base);
    unsigned char* dsm = base + 1024;  // stage s at dsm + s * kStageBytes
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int M = MODE == kDHidden ? R : V;
    const int K = MODE == kDHidden ? V : R;
    const int mt = (M + BM - 1) / BM, ntn = (H + TN - 1) / TN;
    const int ntiles = mt * ntn, nk = (K + KB - 1) / KB;
    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&sb->full[s], 1);
            mbar_init(&sb->xform[s], C::kGroupWarps);
            mbar_init(&sb->empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&sb->acc_full[b], 1);
            mbar_init(&sb->acc_empty[b], 4);
        }
        mbar_init(&sb->drain, 1);
        sb->err = 0;
        sb->timeout_ns = timeout_ns;
        mbar_init_fence();
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                     :: "r"(smem_u32(&sb->tmem_base)), "r"(kTmemCols) : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sb->tmem_base;

    if (warp == 0) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            uint32_t it = 0;
            bool ok = true;
            SegIter<SK> si(ntiles, nk);
            Seg sg;
            while (ok && !*(volatile int*)&sb->err && si.next(sg)) {
                int m0, n0;
                tile_origin(sg.t, mt, ntn, TN, m0, n0);
                for (int kb = sg.kb0; kb < sg.kb1; ++kb) {
                    const int s = (int)(it % S);
                    const uint32_t round = it / S;
                    if (round > 0 && !wait_phase(&sb->empty[s], (round - 1) & 1u, sb, status)) {
                        ok = false;
                        break;
                    }
                    unsigned char* st = dsm + s * C::kStageBytes;
                    const int k0 = kb * KB;
                    // kDWeight: the factors of rows k0 .. k0 + KB - 1 that exist
                    const uint32_t fbytes =
                        MODE == kDWeight ? (uint32_t)min(KB, R - k0) * (uint32_t)sizeof(Fac) : 0u;
                    mbar_expect_tx(&sb->full[s], (uint32_t)(C::kABytes + C::kBBytes) + fbytes);
                    if (MODE == kDHidden) {
                        tma_load_2d(st, &tmX, k0, m0, &sb->full[s]);
                    } else {
                        tma_load_2d(st, &tmX, m0, k0, &sb->full[s]);
                        tma_load_2d(st + kBox, &tmX, m0 + 64, k0, &sb->full[s]);
                        vsd::bulk_g2s(st + C::kABytes + C::kBBytes, fac + k0, fbytes,
                                      &sb->full[s], vsd::policy_evict_last());
                    }
#pragma unroll
                    for (int q = 0; q < 4 * NT; ++q)
                        tma_load_2d(st + C::kABytes + q * kBox, &tmB, n0 + 64 * q, k0,
                                    &sb->full[s]);
                    ++it;
                }
            }
            for (uint32_t j = it > (uint32_t)S ? it - S : 0; j < it; ++j)
                wait_phase_drain(&sb->full[j % S], (j / S) & 1u, timeout_ns);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------ MMA issuer
        if (lane == 0) {
            uint32_t it = 0;
            int lt = 0;
            bool ok = true;
            SegIter<SK> si(ntiles, nk);
            Seg sg;
            for (; ok && !*(volatile int*)&sb->err && si.next(sg); ++lt) {
                const int buf = C::kAccBufs == 2 ? (lt & 1) : 0;
                const uint32_t use = C::kAccBufs == 2 ? ((uint32_t)lt >> 1) : (uint32_t)lt;
                if (use > 0 && !wait_phase(&sb->acc_empty[buf], (use - 1) & 1u, sb, status)) break;
                tc_fence_after();
                const uint32_t d = tmem + (uint32_t)(buf * BN);
                for (int kb = sg.kb0; kb < sg.kb1; ++kb) {
                    const int s = (int)(it % S);
                    if (!wait_phase(&sb->xform[s], (it / S) & 1u, sb, status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a = smem_u32(dsm + s * C::kStageBytes), b = a + C::kABytes;
#pragma unroll
                    for (int k = 0; k < KB / 16; ++k) {
                        // K step of 16: 32 bytes along a K-major row, or two
                        // 8-row K groups (2048 bytes) of an MN-major tile
                        uint64_t ad;
                        if (MODE == kDWeight)
                            ad = sdesc_mn_sw128(a + 2048u * k, kBox);
                        else if (KB == 64)
                            ad = sdesc_sw128(a + 32u * k);
                        else
                            ad = sdesc_sw64(a + 32u * k);
#pragma unroll
                        for (int i = 0; i < NT; ++i)
                            mma_bf16(d + (uint32_t)(i * BN), ad,
                                     sdesc_mn_sw128(b + (uint32_t)(i * 4 * kBox) + 2048u * k, kBox),
                                     kIdesc, (kb != sg.kb0 || k != 0) ? 1u : 0u);
                    }
                    mma_commit(&sb->empty[s]);
                    ++it;
                }
                if (!ok) break;
                mma_commit(&sb->acc_full[buf]);
            }
            mma_commit(&sb->drain);
            wait_phase_drain(&sb->drain, 0, timeout_ns);
        }
    } else if (warp < 2 + kXWarps) {
        // ------------------------------------------------------ the A operand
        // The tile's chunks of 8 elements are shared out by row: kDHidden, tile
        // row rl = tid % 128 (logits row m0 + rl, columns k0 ..); kDWeight,
        // logits row k0 + rl, rl = tid % KB, in box hb = (tid / KB) % 2
        // (columns m0 + 64 hb ..).  Each thread makes kCpt chunks of its row.
        constexpr int kRowChunks = MODE == kDHidden ? KB / 8 : 8;
        constexpr int kGroup = MODE == kDHidden ? 128 : 2 * KB;  // threads covering every row once
        constexpr int kGW = C::kGroupWarps;
        constexpr int kCpt = kGroup * kRowChunks / (32 * kGW);
        static_assert(kCpt >= 1 && kGroup * kRowChunks % (32 * kGW) == 0, "chunk shares");
        constexpr int kRowBytes = MODE == kDHidden ? 2 * KB : 128;
        const int xg = (warp - 2) / kGW;                // this warp's group
        const int tid = threadIdx.x - 64 - 32 * kGW * xg;  // thread within the group
        const int j0 = (tid / kGroup) * kCpt;
        const int rl = MODE == kDHidden ? (tid & 127) : (tid % KB);
        const int hb = MODE == kDHidden ? 0 : ((tid / KB) & 1);
        // 16-byte chunk j of the row sits at chunk j ^ sw (the TMA swizzle)
        const int sw = (MODE == kDHidden && KB == 32) ? ((rl >> 1) & 3) : (rl & 7);
        uint32_t it = 0;
        bool ok = true;
        SegIter<SK> si(ntiles, nk);
        Seg sg;
        while (ok && !*(volatile int*)&sb->err && si.next(sg)) {
            int m0, n0;
            tile_origin(sg.t, mt, ntn, TN, m0, n0);
            Fac f = no_row();
            const KlRec* kl = nullptr;
            if (MODE == kDHidden && m0 + rl < R) {
                f = fac[m0 + rl];
                if (klr) kl = klr + (m0 + rl);
                if (!kl) f.nkl = 0;
            }
            for (int kb = sg.kb0; kb < sg.kb1; ++kb, ++it) {
                const int s = (int)(it % S);
                if (s % C::kGroups != xg) continue;  // another group's stage
                const int k0 = kb * KB;
                unsigned char* A = dsm + s * C::kStageBytes;
                uint4* rowp;
                int vb;
                uint32_t slow = 0;
                if (!wait_phase_warp(&sb->full[s], (it / S) & 1u, sb, status)) {
                    ok = false;
                    break;
                }
                if (MODE == kDHidden) {
                    vb = k0;
                    rowp = reinterpret_cast<uint4*>(A + rl * kRowBytes);
                    if (f.flags) slow = slow_chunks<KB>(f, kl, vb, V);
                } else {
                    // the row's factors came with the stage
                    const Fac* sf = reinterpret_cast<const Fac*>(A + C::kABytes + C::kBBytes);
                    f = k0 + rl < R ? sf[rl] : no_row();
                    kl = (klr && f.flags) ? klr + (k0 + rl) : nullptr;
                    if (!kl) f.nkl = 0;
                    vb = m0 + 64 * hb;
                    rowp = reinterpret_cast<uint4*>(A + hb * kBox + rl * kRowBytes);
                    if (f.flags) slow = slow_chunks<64>(f, kl, vb, V);
                }
#pragma unroll
                for (int jj = 0; jj < kCpt; ++jj) {
                    const int j = j0 + jj;
                    make_chunk(rowp + (j ^ sw), f, c, kl, vb + 8 * j, V, (slow >> j) & 1u);
                }
                // the generic-proxy writes become visible to the tensor cores
                vsd::fence_proxy_async();
                __syncwarp();
                if (lane == 0) mbar_arrive(&sb->xform[s]);
            }
        }
    } else {
        // ------------------------------------------------------ epilogue
        const int q = warp & 3;  // TMEM lanes 32q .. 32q + 31
        int lt = 0;
        SegIter<SK> si(ntiles, nk);
        Seg sg;
        for (; si.next(sg); ++lt) {
            const int buf = C::kAccBufs == 2 ? (lt & 1) : 0;
            const uint32_t use = C::kAccBufs == 2 ? ((uint32_t)lt >> 1) : (uint32_t)lt;
            if (!wait_phase_warp(&sb->acc_full[buf], use & 1u, sb, status)) break;
            tc_fence_after();
            int m0, n0;
            tile_origin(sg.t, mt, ntn, TN, m0, n0);
            // a tile this CTA holds in part: added into the zeroed output
            const bool part = SK && (sg.kb0 != 0 || sg.kb1 != nk);
            const int row = m0 + 32 * q + lane;
            const uint32_t taddr = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * BN);
#pragma unroll 1
            for (int cc = 0; cc < TN / 32; ++cc) {
                uint32_t rg[32];
                tmem_ld32(taddr + 32u * cc, rg);
                const int col = n0 + 32 * cc;
                if (row < M && col < H) {
                    float* o = out + (size_t)row * H + col;
#pragma unroll
                    for (int v4 = 0; v4 < 8; ++v4)
                        if (col + 4 * v4 < H) {
                            if (part)
                                atomicAdd(reinterpret_cast<float4*>(o + 4 * v4),
                                          make_float4(__uint_as_float(rg[4 * v4]),
                                                      __uint_as_float(rg[4 * v4 + 1]),
                                                      __uint_as_float(rg[4 * v4 + 2]),
                                                      __uint_as_float(rg[4 * v4 + 3])));
                            else
                                *reinterpret_cast<uint4*>(o + 4 * v4) =
                                    make_uint4(rg[4 * v4], rg[4 * v4 + 1], rg[4 * v4 + 2],
                                               rg[4 * v4 + 3]);
                        }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sb->acc_empty[buf]);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;"
                     :: "r"(tmem), "r"(kTmemCols) : "memory");
    }
}

}  // namespace vsd_bwd

namespace vsd {

namespace {

#ifndef VSD_BWD_NT
#define VSD_BWD_NT 2
#endif
#ifndef VSD_BWD_STREAM_K
#define VSD_BWD_STREAM_K 1
#endif
#ifndef VSD_BWD_KB_DH
#define VSD_BWD_KB_DH 32
#endif
#ifndef VSD_BWD_KB_DW
#define VSD_BWD_KB_DW 32
#endif

template <int MODE, int NT, int KB>
cudaError_t launch_bwd(const void* logits, const void* bmat, int brows, const vsd_bwd::Fac* fac,
                       const KlRec* klr, float c, int R, int V, int H, float* out, int* status,
                       uint64_t timeout_ns, cudaStream_t s) {
    // (vsd_bwd names qualified: vsd::kThreads is another kernel's block size)
    using vsd_lm::make_map_box;
    CUtensorMap tx, tb;
    // the logits tile: kDHidden one K-major box of KB columns x 128 rows
    // (swizzle as wide as its rows); kDWeight 64-column boxes of KB rows
    const bool okx = MODE == vsd_bwd::kDHidden
                         ? make_map_box(&tx, logits, R, V, KB, vsd_bwd::BM, 2 * KB)
                         : make_map_box(&tx, logits, R, V, 64, KB, 128);
    // B: W [V][H] or hidden [R][H], 64-column boxes of KB rows
    if (!okx || !make_map_box(&tb, bmat, brows, H, 64, KB, 128)) return cudaErrorInvalidValue;
    const size_t smem = vsd_bwd::smem_bytes<MODE, NT, KB>();
    constexpr int BM = vsd_bwd::BM, TN = vsd_bwd::BN * NT;
    const int M = MODE == vsd_bwd::kDHidden ? R : V;
    const long long tiles = (long long)((M + BM - 1) / BM) * ((H + TN - 1) / TN);
    const int sms = device_sm_count();
    const int grid = (int)(tiles < sms ? tiles : sms);
    // Stream-K when whole tiles would leave more than a tenth of the SM time
    // idle (and there are more tiles than SMs, so a share is at least a
    // tile): the output is zeroed first, which costs less than that idle time
    // at these sizes.
    const long long slots = (tiles + sms - 1) / sms * sms;
    const bool sk = VSD_BWD_STREAM_K && tiles > sms && (slots - tiles) * 10 > slots;
    auto kern = sk ? vsd_bwd::k_lmhead_bwd<MODE, NT, KB, true>
                   : vsd_bwd::k_lmhead_bwd<MODE, NT, KB, false>;
    cudaError_t e = ensure_dyn_smem((const void*)kern, smem);
    if (e != cudaSuccess) return e;
    if (sk && (e = cudaMemsetAsync(out, 0, (size_t)M * H * sizeof(float), s)) != cudaSuccess)
        return e;
    kern<<<grid, vsd_bwd::kThreads, smem, s>>>(tx, tb, fac, klr, c, R, V, H, out, status,
                                               timeout_ns);
    return cudaGetLastError();
}

}  // namespace

size_t lmhead_backward_fac_bytes(int R) { return (size_t)R * sizeof(vsd_bwd::Fac); }

cudaError_t lmhead_backward(const void* hidden, const void* weight, const void* logits, int R,
                            int V, int H, float T, const RowRec* rows, const Coef* coef,
                            const KlRec* klr, void* fac_scratch, float* d_hidden,
                            float* d_weight, int* status, uint64_t timeout_ns, cudaStream_t s) {
    const float c = (float)(kLog2e / (double)(T == 0.f ? 1.f : T));  // as the E-step's
    vsd_bwd::Fac* fac = static_cast<vsd_bwd::Fac*>(fac_scratch);
    vsd_bwd::k_rowfac<<<(R + 255) / 256, 256, 0, s>>>(rows, coef, klr, R, fac);
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess && d_hidden)  // G . W
        e = launch_bwd<vsd_bwd::kDHidden, VSD_BWD_NT, VSD_BWD_KB_DH>(
            logits, weight, V, fac, klr, c, R, V, H, d_hidden, status, timeout_ns, s);
    if (e == cudaSuccess && d_weight)  // G^T . hidden
        e = launch_bwd<vsd_bwd::kDWeight, VSD_BWD_NT, VSD_BWD_KB_DW>(
            logits, hidden, R, fac, klr, c, R, V, H, d_weight, status, timeout_ns, s);
    return e;
}

}  // namespace vsd
