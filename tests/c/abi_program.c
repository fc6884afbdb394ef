/*
 * A plain C99 user of libmtdao.so: compiled against include/mtdao.h alone
 * (no CUDA headers, no C++) and linked against the library.  Two modes:
 *
 *   abi_program host
 *       host-only calls (defaults, validation, layout, schedule, half-life
 *       helpers); prints one "key value" line per result.
 *   abi_program run <dir>
 *       reads <dir>/spec.txt ("M T n_tensors numel..."), <dir>/x0.bin
 *       ([n_padded] float32) and <dir>/grads.bin ([T][M][n_padded]
 *       float32), takes T local steps of MT-DAO-Adam (the library's
 *       defaults for N = 2, all periods 4) with the gradients in ordinary
 *       host memory, and writes every state of every replica to
 *       <dir>/states.bin ([n_states][M][n_padded] float32).
 *
 * Exit status 0 on success; any library error is printed and returns 1.
 */
#include <stdio.h>
#include <stdlib.h>

#include "mtdao.h"

#define CHECK(call)                                                                        \
    do {                                                                                   \
        int rc_ = (call);                                                                  \
        if (rc_ != MTDAO_OK) {                                                             \
            fprintf(stderr, "%s failed: %d (%s)\n", #call, rc_, mtdao_last_error(h));      \
            return 1;                                                                      \
        }                                                                                  \
    } while (0)

static int host_mode(void) {
    mtdao_handle h = NULL;
    mtdao_config cfg;
    int64_t numel[3] = {1000, 7, 4096};
    int64_t offsets[3], n_padded = 0;
    double tau = 0.0, saving = 0.0;
    uint32_t mask = 0;
    int64_t t;

    printf("version %d\n", (int)mtdao_version());
    CHECK(mtdao_config_default(&cfg, MTDAO_BASE_ADAM, 2));
    CHECK(mtdao_config_validate(&cfg, 4));
    printf("num_states %d\n", (int)mtdao_num_states(&cfg));
    CHECK(mtdao_plan_layout(numel, 3, offsets, &n_padded));
    printf("layout %lld %lld %lld %lld\n", (long long)offsets[0], (long long)offsets[1],
           (long long)offsets[2], (long long)n_padded);
    cfg.period_x = 6;
    cfg.period_u[0] = 2;
    cfg.period_u[1] = 3;
    cfg.period_v = 4;
    printf("masks");
    for (t = 0; t < 12; ++t) {
        CHECK(mtdao_due_mask(&cfg, t, &mask));
        printf(" %u", (unsigned)mask);
    }
    printf("\n");
    CHECK(mtdao_half_life(0.999, &tau));
    printf("half_life %.17g\n", tau);
    CHECK(mtdao_config_half_life_periods(&cfg, 32));
    printf("half_life_periods %lld %lld %lld %lld\n", (long long)cfg.period_x,
           (long long)cfg.period_u[0], (long long)cfg.period_u[1], (long long)cfg.period_v);
    CHECK(mtdao_comm_reduction(&cfg, &saving));
    printf("comm_reduction %.17g\n", saving);
    cfg.beta1[0] = 1.0;                                  /* out of range: must be rejected */
    printf("invalid %d\n", mtdao_config_validate(&cfg, 4));
    return 0;
}

static float *read_floats(const char *dir, const char *name, size_t count) {
    char path[4096];
    FILE *f;
    float *buf = (float *)malloc(count * sizeof(float));
    snprintf(path, sizeof path, "%s/%s", dir, name);
    f = fopen(path, "rb");
    if (buf == NULL || f == NULL || fread(buf, sizeof(float), count, f) != count) {
        fprintf(stderr, "cannot read %s\n", path);
        if (f) fclose(f);
        free(buf);
        return NULL;
    }
    fclose(f);
    return buf;
}

static int run_mode(const char *dir) {
    mtdao_handle h = NULL;
    mtdao_config cfg;
    int M = 0, T = 0, n_tensors = 0, k, m, s, t, n_states;
    int64_t numel[64], offsets[64], n_padded = 0;
    float *x0, *grads, *out;
    char path[4096];
    FILE *f;
    uint32_t mask = 0;

    snprintf(path, sizeof path, "%s/spec.txt", dir);
    f = fopen(path, "r");
    if (f == NULL || fscanf(f, "%d %d %d", &M, &T, &n_tensors) != 3 || n_tensors < 1 || n_tensors > 64) {
        fprintf(stderr, "bad spec\n");
        return 1;
    }
    for (k = 0; k < n_tensors; ++k) {
        long long v;
        if (fscanf(f, "%lld", &v) != 1) return 1;
        numel[k] = v;
    }
    fclose(f);

    CHECK(mtdao_config_default(&cfg, MTDAO_BASE_ADAM, 2));
    cfg.period_x = cfg.period_u[0] = cfg.period_u[1] = cfg.period_v = 4;
    CHECK(mtdao_plan_layout(numel, n_tensors, offsets, &n_padded));
    CHECK(mtdao_create(&cfg, M, numel, n_tensors, NULL, &h));
    n_states = mtdao_num_states(&cfg);

    x0 = read_floats(dir, "x0.bin", (size_t)n_padded);
    grads = read_floats(dir, "grads.bin", (size_t)T * M * n_padded);
    out = (float *)malloc((size_t)n_states * M * n_padded * sizeof(float));
    if (x0 == NULL || grads == NULL || out == NULL) return 1;

    for (m = 0; m < M; ++m) CHECK(mtdao_copy_state_from_host(h, 0, m, x0));   /* x_0 on every worker */
    for (t = 0; t < T; ++t) {
        CHECK(mtdao_sync_due(h, &mask));
        CHECK(mtdao_step_host(h, grads + (size_t)t * M * n_padded, MTDAO_F32, 1e-3, mask));
    }
    for (s = 0; s < n_states; ++s)
        for (m = 0; m < M; ++m)
            CHECK(mtdao_copy_state_to_host(h, s, m, out + ((size_t)s * M + m) * n_padded));
    printf("steps %lld\n", (long long)mtdao_get_step(h));
    mtdao_destroy(h);

    snprintf(path, sizeof path, "%s/states.bin", dir);
    f = fopen(path, "wb");
    if (f == NULL || fwrite(out, sizeof(float), (size_t)n_states * M * n_padded, f) !=
                         (size_t)n_states * M * n_padded)
        return 1;
    fclose(f);
    free(x0);
    free(grads);
    free(out);
    return 0;
}

int main(int argc, char **argv) {
    if (argc >= 2 && argv[1][0] == 'h') return host_mode();
    if (argc >= 3 && argv[1][0] == 'r') return run_mode(argv[2]);
    fprintf(stderr, "usage: %s host | run <dir>\n", argv[0]);
    return 2;
}
