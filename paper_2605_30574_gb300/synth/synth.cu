// Device twin of the seeded synthetic-input generator (host twin: host.py).
//
// Every value is a pure function of its logical coordinates:
//   stream state x0 = mix(seed * 256 + stream + GAMMA)
//   draw(i)         = mix(x0 + (i + 1) * GAMMA)          (splitmix64, Steele,
//                     Lea & Flood 2014; mix = the 64-bit finaliser)
//   z               = f32(sum of the four 16-bit fields - 131070) * f32(1/37837.2272...)
//   value           = bf16_rne(f32(z * mult))
// with the element index = row-major linear index of the coordinates (see
// host.py for the stream list).  Fills whole device stores; holds none of the
// splice or attention arithmetic.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;
constexpr uint64_t kMix1 = 0xBF58476D1CE4E5B9ull;
constexpr uint64_t kMix2 = 0x94D049BB133111EBull;
constexpr uint32_t kNormalScaleBits = 0x37DDB3D7u;
constexpr int kCenter = 131070;

enum : int {
    S_Q = 1, S_KSUF = 2, S_VSUF = 3, S_KCLEAN = 4, S_VCLEAN = 5,
    S_KFILL = 6, S_VFILL = 7, S_KNOISE = 8, S_VNOISE = 9, S_PMASK = 10
};
enum : int { K_ZERO = 0, K_BLANK = 1, K_SAME = 2, K_DIFF_ALGO = 3, K_DIFF_FAMILY = 4 };

__host__ __device__ inline uint64_t mix(uint64_t z) {
    z = (z ^ (z >> 30)) * kMix1;
    z = (z ^ (z >> 27)) * kMix2;
    return z ^ (z >> 31);
}

__host__ __device__ inline uint64_t stream_state(uint64_t seed, int stream) {
    return mix(seed * 256ull + uint64_t(stream) + kGamma);
}

__device__ inline uint64_t draw(uint64_t x0, uint64_t idx) { return mix(x0 + (idx + 1ull) * kGamma); }

__device__ inline uint16_t bf16_bits(float f) {
    const __nv_bfloat16 b = __float2bfloat16_rn(f);
    return *reinterpret_cast<const uint16_t*>(&b);
}

__device__ inline float bf16_value(uint16_t u) { return __uint_as_float(uint32_t(u) << 16); }

__device__ inline uint16_t normal_bf16(uint64_t x0, uint64_t idx, float mult) {
    const uint64_t u = draw(x0, idx);
    const int c = int(u & 0xffff) + int((u >> 16) & 0xffff) + int((u >> 32) & 0xffff) + int(u >> 48) - kCenter;
    float z = __fmul_rn(float(c), __uint_as_float(kNormalScaleBits));
    if (mult != 1.0f) z = __fmul_rn(z, mult);
    return bf16_bits(z);
}

struct Streams {
    uint64_t x[11];
};

Streams make_streams(uint64_t seed) {
    Streams s;
    for (int i = 0; i < 11; ++i) s.x[i] = stream_state(seed, i);
    return s;
}

__global__ void normal_kernel(uint64_t x0, uint64_t idx0, long n, float mult, uint16_t* out) {
    for (long i = long(blockIdx.x) * blockDim.x + threadIdx.x; i < n; i += long(gridDim.x) * blockDim.x)
        out[i] = normal_bf16(x0, idx0 + uint64_t(i), mult);
}

// Clean prompt-span store [Pl][N][Hkv][Tp][d] for prompts p0 .. p0 + Pl - 1.
__global__ void clean_kernel(Streams st, int p0, int Pl, int Pt, int N, int Hkv, int Tp, int d,
                             uint16_t* k, uint16_t* v) {
    const long total = long(Pl) * N * Hkv * Tp * d;
    for (long i = long(blockIdx.x) * blockDim.x + threadIdx.x; i < total; i += long(gridDim.x) * blockDim.x) {
        const long row = i / d;                 // ((pl * N + l) * Hkv + h) * Tp + j
        const int j = int(row % Tp);
        const long pl = row / (long(N) * Hkv * Tp);
        const uint64_t idx = uint64_t(i) + uint64_t(p0) * uint64_t(N) * Hkv * Tp * d;
        (void)Pt;
        k[i] = normal_bf16(st.x[S_KCLEAN], idx, j == 0 ? 20.0f : 1.0f);
        v[i] = normal_bf16(st.x[S_VCLEAN], idx, 1.0f);
        (void)pl;
    }
}

// Donor store [Pl][Dst][N][Hkv][Tp][d] (stored slots in slot order).
__global__ void donor_kernel(Streams st, int p0, int Pl, int Dslots, int Dst, const int* stored_slot,
                             const int* kinds, const uint32_t* thr24, int N, int Hkv, int Tp, int d,
                             int sc_head, int sc_tail, uint16_t* k, uint16_t* v) {
    const long per_slot = long(N) * Hkv * Tp * d;
    const long total = long(Pl) * Dst * per_slot;
    for (long i = long(blockIdx.x) * blockDim.x + threadIdx.x; i < total; i += long(gridDim.x) * blockDim.x) {
        const long inner = i % per_slot;       // ((l * Hkv + h) * Tp + j) * d + c
        const long ps = i / per_slot;           // pl * Dst + st
        const int sidx = int(ps % Dst);
        const int p = p0 + int(ps / Dst);
        const int slot = stored_slot[sidx];
        const int kind = kinds[slot];
        const int j = int((inner / d) % Tp);
        const uint64_t cidx = uint64_t(p) * uint64_t(per_slot) + uint64_t(inner);
        const uint16_t ck = normal_bf16(st.x[S_KCLEAN], cidx, j == 0 ? 20.0f : 1.0f);
        const uint16_t cv = normal_bf16(st.x[S_VCLEAN], cidx, 1.0f);
        const bool scaffold = j < sc_head || j >= Tp - sc_tail;
        const uint64_t didx = (uint64_t(p) * Dslots + slot) * uint64_t(per_slot) + uint64_t(inner);
        uint16_t ok = ck, ov = cv;
        if (!scaffold) {
            if (kind == K_BLANK || kind == K_DIFF_FAMILY) {
                ok = normal_bf16(st.x[S_KFILL], didx, 1.0f);
                ov = normal_bf16(st.x[S_VFILL], didx, 1.0f);
            } else {
                const uint64_t u = draw(st.x[S_PMASK], (uint64_t(p) * Dslots + slot) * Tp + j);
                if ((u >> 40) < uint64_t(thr24[slot])) {
                    const float nk = __fmul_rn(bf16_value(normal_bf16(st.x[S_KNOISE], didx, 1.0f)), 0.5f);
                    const float nv = __fmul_rn(bf16_value(normal_bf16(st.x[S_VNOISE], didx, 1.0f)), 0.5f);
                    ok = bf16_bits(__fadd_rn(bf16_value(ck), nk));
                    ov = bf16_bits(__fadd_rn(bf16_value(cv), nv));
                }
            }
        }
        k[i] = ok;
        v[i] = ov;
    }
}

// Generated-span store [Bl][N][Hkv][T][d] of sequences s0 .. s0 + Bl - 1, all T slots.
__global__ void suffix_kernel(Streams st, long s0, int Bl, int N, int Hkv, int T, int d, uint16_t* k,
                              uint16_t* v) {
    const long total = long(Bl) * N * Hkv * T * d;
    const uint64_t base = uint64_t(s0) * uint64_t(N) * Hkv * T * d;
    for (long i = long(blockIdx.x) * blockDim.x + threadIdx.x; i < total; i += long(gridDim.x) * blockDim.x) {
        k[i] = normal_bf16(st.x[S_KSUF], base + uint64_t(i), 1.0f);
        v[i] = normal_bf16(st.x[S_VSUF], base + uint64_t(i), 1.0f);
    }
}

// This step's generated K/V [Bl][Hkv][d] at layer l (= generated-span slot t - 1).
__global__ void new_kv_kernel(Streams st, long s0, int Bl, int N, int Hkv, int T, int d, int l, int t,
                              uint16_t* k, uint16_t* v) {
    const long total = long(Bl) * Hkv * d;
    for (long i = long(blockIdx.x) * blockDim.x + threadIdx.x; i < total; i += long(gridDim.x) * blockDim.x) {
        const int c = int(i % d);
        const long bh = i / d;
        const int h = int(bh % Hkv);
        const long s = s0 + bh / Hkv;
        const uint64_t idx = (((uint64_t(s) * N + l) * Hkv + h) * T + (t - 1)) * d + c;
        k[i] = normal_bf16(st.x[S_KSUF], idx, 1.0f);
        v[i] = normal_bf16(st.x[S_VSUF], idx, 1.0f);
    }
}

// Queries [Bl][Hq][d] at step t, layer l.
__global__ void q_kernel(Streams st, long s0, int Bl, int N, int Hq, int T, int d, int l, int t, float qmult,
                         uint16_t* q) {
    const long total = long(Bl) * Hq * d;
    for (long i = long(blockIdx.x) * blockDim.x + threadIdx.x; i < total; i += long(gridDim.x) * blockDim.x) {
        const int c = int(i % d);
        const long bh = i / d;
        const int hq = int(bh % Hq);
        const long s = s0 + bh / Hq;
        const uint64_t idx = (((uint64_t(s) * (T + 1) + t) * N + l) * Hq + hq) * d + c;
        q[i] = normal_bf16(st.x[S_Q], idx, qmult);
    }
}

unsigned grid_for(long n) {
    long b = (n + 255) / 256;
    if (b > 152L * 64) b = 152L * 64;
    return unsigned(b < 1 ? 1 : b);
}

}  // namespace

extern "C" {

int synth_normal(uint64_t seed, int stream, uint64_t idx0, long n, float mult, uint16_t* out, void* s) {
    normal_kernel<<<grid_for(n), 256, 0, (cudaStream_t)s>>>(stream_state(seed, stream), idx0, n, mult, out);
    return int(cudaGetLastError());
}

int synth_fill_clean(uint64_t seed, int p0, int Pl, int Pt, int N, int Hkv, int Tp, int d, uint16_t* k,
                     uint16_t* v, void* s) {
    const long n = long(Pl) * N * Hkv * Tp * d;
    clean_kernel<<<grid_for(n), 256, 0, (cudaStream_t)s>>>(make_streams(seed), p0, Pl, Pt, N, Hkv, Tp, d, k, v);
    return int(cudaGetLastError());
}

// kinds / thr24: [Dslots] on the host; copied into a small device buffer
// owned by this call (synchronous).
int synth_fill_donor(uint64_t seed, int p0, int Pl, int Dslots, const int* kinds_h, const uint32_t* thr24_h,
                     int N, int Hkv, int Tp, int d, int sc_head, int sc_tail, uint16_t* k, uint16_t* v,
                     void* s) {
    int stored[256];
    int Dst = 0;
    for (int i = 0; i < Dslots && i < 256; ++i)
        if (kinds_h[i] != K_ZERO) stored[Dst++] = i;
    if (Dst == 0) return 0;
    int* buf = nullptr;
    cudaError_t e = cudaMalloc(&buf, sizeof(int) * (Dst + 2 * Dslots));
    if (e != cudaSuccess) return int(e);
    cudaMemcpy(buf, stored, sizeof(int) * Dst, cudaMemcpyHostToDevice);
    cudaMemcpy(buf + Dst, kinds_h, sizeof(int) * Dslots, cudaMemcpyHostToDevice);
    cudaMemcpy(buf + Dst + Dslots, thr24_h, sizeof(int) * Dslots, cudaMemcpyHostToDevice);
    const long n = long(Pl) * Dst * N * Hkv * Tp * d;
    donor_kernel<<<grid_for(n), 256, 0, (cudaStream_t)s>>>(make_streams(seed), p0, Pl, Dslots, Dst, buf, buf + Dst,
                                                          reinterpret_cast<const uint32_t*>(buf + Dst + Dslots),
                                                          N, Hkv, Tp, d, sc_head, sc_tail, k, v);
    e = cudaGetLastError();
    cudaStreamSynchronize((cudaStream_t)s);
    cudaFree(buf);
    return int(e);
}

int synth_fill_suffix(uint64_t seed, long s0, int Bl, int N, int Hkv, int T, int d, uint16_t* k, uint16_t* v,
                      void* s) {
    const long n = long(Bl) * N * Hkv * T * d;
    suffix_kernel<<<grid_for(n), 256, 0, (cudaStream_t)s>>>(make_streams(seed), s0, Bl, N, Hkv, T, d, k, v);
    return int(cudaGetLastError());
}

int synth_fill_new_kv(uint64_t seed, long s0, int Bl, int N, int Hkv, int T, int d, int l, int t, uint16_t* k,
                      uint16_t* v, void* s) {
    const long n = long(Bl) * Hkv * d;
    new_kv_kernel<<<grid_for(n), 256, 0, (cudaStream_t)s>>>(make_streams(seed), s0, Bl, N, Hkv, T, d, l, t, k, v);
    return int(cudaGetLastError());
}

int synth_fill_q(uint64_t seed, long s0, int Bl, int N, int Hq, int T, int d, int l, int t, float qmult,
                 uint16_t* q, void* s) {
    const long n = long(Bl) * Hq * d;
    q_kernel<<<grid_for(n), 256, 0, (cudaStream_t)s>>>(make_streams(seed), s0, Bl, N, Hq, T, d, l, t, qmult, q);
    return int(cudaGetLastError());
}

}  // extern "C"
