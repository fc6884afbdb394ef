// synth_dev.cu -- seeded, counter-based synthetic inputs generated on the GPU.
//
// Input plumbing for the tests and the benchmark, not part of the optimizer:
// it holds none of the method's arithmetic.  It implements, independently of
// the numpy generator in generators.py, the same definition:
//
//   mix(z): SplitMix64 output function (Steele, Lea & Flood, OOPSLA 2014):
//           z += 0x9E3779B97F4A7C15; z = (z ^ z>>30) * 0xBF58476D1CE4E5B9;
//           z = (z ^ z>>27) * 0x94D049BB133111EB; z ^= z>>31
//   key    = mix(mix(mix(seed ^ stream) ^ m) ^ t)   stream 1 = gradients, 2 = x_0
//   e      = mix(key ^ i)                           i = padded element index
//   word_k = mix(e ^ k)
//   Z(k0)  = float(2*S - 786420) * 2^-17, S = sum of the twelve 16-bit lanes
//            of word_k0 .. word_k0+2 (Irwin-Hall normal, exact in fp32)
//   kinds  : normal g = Z(0)*sigma;  student_t3 g = (Z(0)/sqrt(max(
//            ((Z(3)^2 + Z(6)^2) + Z(9)^2)/3, 2^-20))) * sigma;
//            normal_outliers g = Z(0)*sigma, times 100 when the low 32 bits of
//            word_12 are below 42949673
//   bf16   : round-to-nearest-even of the fp32 bits; padding elements are 0.
// Every floating-point step is a single IEEE round-to-nearest operation
// (explicit __f*_rn intrinsics, so nothing is contracted into an FMA), which
// makes the output bit-identical to the host generator.
#include <cuda_runtime.h>
#include <cstdint>

namespace {

__device__ __forceinline__ uint64_t mix(uint64_t z) {
    z += 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ float irwin_hall_normal(uint64_t e, uint64_t k0) {
    int64_t s = 0;
    for (uint64_t k = k0; k < k0 + 3; ++k) {
        const uint64_t w = mix(e ^ k);
        s += static_cast<int64_t>(w & 0xFFFFull) + static_cast<int64_t>((w >> 16) & 0xFFFFull) +
             static_cast<int64_t>((w >> 32) & 0xFFFFull) + static_cast<int64_t>((w >> 48) & 0xFFFFull);
    }
    return __fmul_rn(__ll2float_rn(2 * s - 786420), 7.62939453125e-06f);   // 2^-17
}

__device__ bool inside_tensor(int64_t i, const int64_t *off, const int64_t *num, int nt) {
    int lo = 0, hi = nt - 1;
    while (lo < hi) {                       // last tensor with offset <= i
        const int mid = (lo + hi + 1) >> 1;
        if (off[mid] <= i) lo = mid; else hi = mid - 1;
    }
    return i >= off[lo] && i < off[lo] + num[lo];
}

__global__ void fill_kernel(void *out, int bf16, int kind, uint64_t seed, uint64_t stream, int M,
                            int64_t n, int64_t t, float sigma, const int64_t *off, const int64_t *num,
                            int nt) {
    const int64_t total = static_cast<int64_t>(M) * n;
    for (int64_t f = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; f < total;
         f += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t m = f / n, i = f - m * n;
        float g = 0.0f;
        if (inside_tensor(i, off, num, nt)) {
            const uint64_t key = mix(mix(mix(seed ^ stream) ^ static_cast<uint64_t>(m)) ^
                                     static_cast<uint64_t>(t));
            const uint64_t e = mix(key ^ static_cast<uint64_t>(i));
            const float z0 = irwin_hall_normal(e, 0);
            if (kind == 1) {
                const float z1 = irwin_hall_normal(e, 3), z2 = irwin_hall_normal(e, 6),
                            z3 = irwin_hall_normal(e, 9);
                float a = __fmul_rn(z1, z1);
                a = __fadd_rn(a, __fmul_rn(z2, z2));
                a = __fadd_rn(a, __fmul_rn(z3, z3));
                a = __fdiv_rn(a, 3.0f);
                a = fmaxf(a, 9.5367431640625e-07f);                         // 2^-20
                g = __fmul_rn(__fdiv_rn(z0, __fsqrt_rn(a)), sigma);
            } else {
                g = __fmul_rn(z0, sigma);
                if (kind == 2) {
                    const uint32_t low = static_cast<uint32_t>(mix(e ^ 12ull) & 0xFFFFFFFFull);
                    if (low < 42949673u) g = __fmul_rn(g, 100.0f);
                }
            }
        }
        if (bf16) {
            uint32_t b = __float_as_uint(g);
            b += 0x7FFFu + ((b >> 16) & 1u);
            static_cast<uint16_t *>(out)[f] = static_cast<uint16_t>(b >> 16);
        } else {
            static_cast<float *>(out)[f] = g;
        }
    }
}

// Gradient of a toy objective at each worker's current parameters, plus
// noise sigma * Z (Z from stream 3: key(seed, 3, m, t), element i, word 0).
//   kind 0, quadratic  f = sum_i lambda_i x_i^2 / 2:   g_i = lambda_i x_i
//   kind 1, Rosenbrock f = sum_k (1 - a_k)^2 + 100 (b_k - a_k^2)^2 over the
//           pairs (a_k, b_k) = (x_2k, x_2k+1):
//           g_a = 2 (a - 1) - 400 a (b - a^2),   g_b = 200 (b - a^2)
// Elements at or beyond n_real are padding and get 0.
__global__ void toy_grad_kernel(int kind, const float *x, float *g, int M, int64_t n, int64_t n_real,
                                uint64_t seed, int64_t t, float sigma, const float *lam) {
    const int64_t total = static_cast<int64_t>(M) * n;
    for (int64_t f = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; f < total;
         f += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t m = f / n, i = f - m * n;
        float out = 0.0f;
        if (i < n_real) {
            const uint64_t key = mix(mix(mix(seed ^ 3ull) ^ static_cast<uint64_t>(m)) ^
                                     static_cast<uint64_t>(t));
            const float z = irwin_hall_normal(mix(key ^ static_cast<uint64_t>(i)), 0);
            // evaluated in double (toy sizes make that free) so that the
            // objective's own rounding -- b - a^2 cancels near the valley --
            // stays far below the optimizer's
            double grad;
            if (kind == 0) {
                grad = static_cast<double>(lam[i]) * static_cast<double>(x[f]);
            } else {
                const int64_t base = f - (i & 1);
                const double a = x[base], b = x[base + 1];
                const double r = b - a * a;
                grad = (i & 1) ? 200.0 * r : 2.0 * (a - 1.0) - 400.0 * a * r;
            }
            out = static_cast<float>(grad + static_cast<double>(sigma) * static_cast<double>(z));
        }
        g[f] = out;
    }
}

}  // namespace

// Toy-objective gradients for the M workers' parameters x_dev ([M][n_padded]
// fp32, e.g. state 0 of an MT-DAO handle) into g_dev ([M][n_padded] fp32).
// kind 0: quadratic with per-element curvature lam_dev ([n_padded]);
// kind 1: Rosenbrock pairs (n_real even).  Returns a cudaError_t value.
extern "C" int synth_toy_grad(int kind, const float *x_dev, float *g_dev, int M, int64_t n_padded,
                              int64_t n_real, uint64_t seed, int64_t t, float sigma,
                              const float *lam_dev, void *cuda_stream) {
    if (x_dev == nullptr || g_dev == nullptr || M < 1 || n_padded < 1 || n_real > n_padded ||
        (kind == 0 && lam_dev == nullptr) || (kind == 1 && (n_real & 1)) || kind < 0 || kind > 1)
        return cudaErrorInvalidValue;
    const int64_t total = static_cast<int64_t>(M) * n_padded;
    int64_t grid = (total + 255) / 256;
    if (grid > 4096) grid = 4096;
    toy_grad_kernel<<<static_cast<unsigned>(grid), 256, 0, static_cast<cudaStream_t>(cuda_stream)>>>(
        kind, x_dev, g_dev, M, n_padded, n_real, seed, t, sigma, lam_dev);
    return static_cast<int>(cudaGetLastError());
}

// Fill out_dev[M][n_padded] (f32, or bf16 when bf16 != 0) for step t.
// kind: 0 normal, 1 student_t3, 2 normal_outliers.  stream_id: 1 gradients,
// 2 initial parameters (then use M = 1, t = 0).  offsets/numels: device
// arrays of the tensor layout.  Returns a cudaError_t value.
extern "C" int synth_fill(void *out_dev, int bf16, int kind, uint64_t seed, uint64_t stream_id, int M,
                          int64_t n_padded, int64_t t, float sigma, const int64_t *offsets_dev,
                          const int64_t *numels_dev, int n_tensors, void *cuda_stream) {
    if (out_dev == nullptr || M < 1 || n_padded < 1 || n_tensors < 1) return cudaErrorInvalidValue;
    int dev = 0, sms = 1;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t total = static_cast<int64_t>(M) * n_padded;
    int64_t grid = (total + 255) / 256;
    if (grid > static_cast<int64_t>(sms) * 8) grid = static_cast<int64_t>(sms) * 8;
    fill_kernel<<<static_cast<unsigned>(grid), 256, 0, static_cast<cudaStream_t>(cuda_stream)>>>(
        out_dev, bf16, kind, seed, stream_id, M, n_padded, t, sigma, offsets_dev, numels_dev, n_tensors);
    return static_cast<int>(cudaGetLastError());
}
